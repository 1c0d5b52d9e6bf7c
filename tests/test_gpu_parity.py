"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.

* hash locations: bit-exact;
* pooled forward: within 1e-6 of sum|terms| (bit-exact on dyadic inputs);
* gradient (Algorithm 1 dense branch): within 1e-5 of sum|contributions|;
* updated shared array and Adagrad accumulator: the derived bounds in gpu_util.

Sizes: small cases that span many thread blocks and a ragged tail, then the
named workloads at full size (tiny, Criteo-Kaggle, Criteo-TB, multi-hot
contention, the compression sweep), in the default launch configuration that
bench.py times.
"""
import numpy as np
import pytest

from paper_2207_10731_gb300 import binding, workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


def _batch_cuda(w):
    return gu.cuda(w.indices), gu.cuda(w.offsets)


def _abs_pool(o, w_host, w):
    out, _ = o.forward(np.abs(w_host), w.indices, w.offsets, w.B)
    return out


# --------------------------------------------------------------------------
# hash (row a2): bit-exact
LOC_CASES = [
    dict(name="tiny"),
    dict(name="kaggle"),
    dict(name="tb", B=4096),
    dict(name="multihot", B=512),
    dict(name="tiny", G=1),                 # paper-literal offsets, scalar path
    dict(name="tiny", Z=1, G=1),            # HashedNet (Z = 1)
    dict(name="kaggle", Z=3, G=2, B=300),   # odd chunk, ragged tail
]


@pytest.mark.parametrize("case", LOC_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_locations_bit_exact(case):
    case = dict(case)
    w = wl.make_workload(case.pop("name"), grad="none", **case)
    h, o = gu.make_pair(w)
    idx, off = _batch_cuda(w)
    got = gu.host(h.compute_locations(idx, off, w.B))
    want, bad = o.locations(w.indices, w.offsets, w.B)
    assert bad == -1
    np.testing.assert_array_equal(got, want)
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()


def test_locations_beyond_32_bits():
    # M > 2^32 elements: block starts need 64-bit offsets.
    w = wl.make_workload("tb", B=2048, M=(1 << 33), grad="none")
    h = binding.PSS(w.cards, dim=w.d, M=w.M, Z=w.Z, G=w.G, seed=0)
    from oracle import OraclePSS
    o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=0)
    got = gu.host(h.compute_locations(*_batch_cuda(w), w.B))
    want, _ = o.locations(w.indices, w.offsets, w.B)
    np.testing.assert_array_equal(got, want)
    assert got.max() > (1 << 32)
    h.close()


# --------------------------------------------------------------------------
# forward (row a3)
FWD_CASES = [
    dict(name="tiny"),
    dict(name="kaggle"),
    dict(name="tb", B=8192),
    dict(name="multihot", B=2048),
    dict(name="multihot", B=777, bag=("uniform", 0, 6)),      # empty bags, ragged tail
    dict(name="tiny", G=1),
    dict(name="tiny", Z=1, G=1),
    dict(name="kaggle", Z=3, G=2, B=300),
    dict(name="tb", B=1000, d=200, Z=32),                    # two columns per lane
    dict(name="tb", B=600, d=384, Z=64, G=8),                # three 16-byte columns per lane
    dict(name="tb", B=500, d=10, Z=4, G=4),                  # d not a multiple of 4
]


def _wl(case):
    case = dict(case)
    name = case.pop("name")
    over = {k: case.pop(k) for k in ("bag", "d") if k in case}
    return wl.make_workload(name, **case, **over)


@pytest.mark.parametrize("case", FWD_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_forward_parity(case):
    w = _wl(case)
    h, o = gu.make_pair(w)
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, bad = o.forward(w.w0, w.indices, w.offsets, w.B)
    assert bad == -1
    gu.check_forward(out, ref, _abs_pool(o, w.w0, w))
    h.close()


@pytest.mark.parametrize("name,B", [("tiny", 256), ("kaggle", 2048), ("multihot", 1024)])
def test_forward_dyadic_bit_exact(name, B):
    w = wl.make_workload(name, B=B, w0="dyadic")
    h, o = gu.make_pair(w)
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, _ = o.forward(w.w0, w.indices, w.offsets, w.B)
    np.testing.assert_array_equal(out, ref)
    h.close()


# --------------------------------------------------------------------------
# gradient (row a4): lr = 0 capture through pss_backward_grad
PATHS = {"auto": binding.PATH_AUTO, "atomic": binding.PATH_ATOMIC, "sorted": binding.PATH_SORTED}


def _set_path(h, path):
    """Select a backward path by name: "sorted" leaves the sort scope automatic,
    "sorted-local" and "sorted-global" force the segment-local sort (where
    the chunks tile the rows) or one sort over all pairs.  Returns the PATH_*
    value."""
    if path in ("sorted-global", "sorted-local"):
        h.set_option(binding.OPT_SORT_SCOPE,
                     binding.SORT_GLOBAL if path == "sorted-global" else binding.SORT_LOCAL)
        path = "sorted"
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS[path])
    return PATHS[path]


@pytest.mark.parametrize("path", list(PATHS) + ["sorted-global", "sorted-local"])
@pytest.mark.parametrize("case", FWD_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_grad_parity(case, path):
    w = _wl(case)
    h, o = gu.make_pair(w)
    want = _set_path(h, path)
    h.forward(*_batch_cuda(w), w.B)
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    ref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, ref, A)
    # total mass: sum over bags of |bag| * sum of its upstream gradient row
    lengths = np.diff(w.offsets).reshape(w.T, w.B)
    rows = w.grad_out.reshape(w.B, w.T, w.d).astype(np.float64).sum(axis=2)
    mass = float((lengths.T * rows).sum())
    assert abs(g.astype(np.float64).sum() - mass) <= 1e-5 * A.sum() + 1e-6
    if path != "auto":
        assert h.info()["last_path"] == want
    h.close()


@pytest.mark.parametrize("path", ["atomic", "sorted", "sorted-deterministic"])
def test_grad_single_hot_id_and_repeated_backward(path):
    # Every bag of every table holds id 0, so each table's J buckets collect
    # all B contributions (the most skewed batch there is); B is not a
    # multiple of any segment or tile size.  A second backward of the same
    # batch must give the same gradient.
    w = wl.make_workload("tb", B=5003)
    w.indices[:] = 0
    h, o = gu.make_pair(w)
    if path == "sorted-deterministic":
        # every bucket's run fills about a thousand reduce tasks: the window
        # reduce's boundary combine adds them all up
        h.set_option(binding.OPT_DETERMINISTIC, 1)
        path = "sorted"
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS[path])
    h.forward(*_batch_cuda(w), w.B)
    go = gu.cuda(w.grad_out)
    g1 = gu.host(h.backward_grad(go))
    g2 = gu.host(h.backward_grad(go))
    ref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g1, ref, A)
    gu.check_grad(g2, ref, A)
    assert h.info()["last_path"] == PATHS[path]
    h.close()


def test_grad_dyadic_and_all_ones_exact():
    for grad in ("dyadic", "ones"):
        w = wl.make_workload("kaggle", B=1024, grad=grad, w0="dyadic")
        h, o = gu.make_pair(w)
        h.forward(*_batch_cuda(w), w.B)
        g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
        ref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
        np.testing.assert_array_equal(g.astype(np.float64), ref)
        h.close()


# --------------------------------------------------------------------------
# fused backward + optimizer step (rows a4, a5)
STEP_CASES = [
    dict(name="tiny"),                                  # SGD lr 0.1
    dict(name="kaggle"),                                # Adagrad
    dict(name="tb", B=8192),                            # Adagrad
    dict(name="multihot", B=2048),                      # SGD, contention
    dict(name="kaggle", opt="sgd"),
    dict(name="tiny", opt="adagrad", lr=0.05),
    dict(name="multihot", B=777, bag=("uniform", 0, 6), opt="adagrad"),
    dict(name="tiny", G=1, opt="adagrad"),
    dict(name="tiny", Z=1, G=1),
]


def _run_step(w, h, o, wcur, Gcur, batch):
    idx, off, go = batch
    B = (off.shape[0] - 1) // w.T
    h.forward(gu.cuda(idx), gu.cuda(off), B)
    h.backward_update(gu.cuda(go), w.lr)
    wg, Gg = h.get_state()
    w2, G2, g32 = o.step(wcur, Gcur, idx, off, B, go, w.opt, w.lr, w.eps)
    A = o.grad(idx, off, B, np.abs(go))
    return gu.host(wg), (gu.host(Gg) if Gg is not None else None), w2, G2, g32, A


@pytest.mark.parametrize("path", list(PATHS) + ["sorted-global", "sorted-local"])
@pytest.mark.parametrize("case", STEP_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_step_parity_three_steps(case, path):
    case = dict(case)
    opt = case.pop("opt", None)
    lr = case.pop("lr", None)
    w = _wl(case)
    if opt:
        w.opt = opt
    if lr:
        w.lr = lr
    h, o = gu.make_pair(w)
    _set_path(h, path)
    wcur = w.w0.copy()
    Gcur = np.zeros(w.M, dtype=np.float32)
    cfg = wl.CONFIGS[case["name"]]
    for step in range(3):
        if step == 0:
            batch = (w.indices, w.offsets, w.grad_out)
        else:
            batch = wl.make_batch(w.cards, w.B, w.d, case.get("bag", cfg["bag"]), cfg["ids"],
                                  seed=w.seed, batch=step)
        wg, Gg, wcur_next, Gnext, g32, A = _run_step(w, h, o, wcur, Gcur, batch)
        if w.opt == "sgd":
            gu.check_sgd(wg, wcur_next, A, w.lr, what=f"sgd step {step}")
        else:
            gu.check_adagrad(wg, Gg, wcur_next, Gnext, g32, A, w.lr, what=f"adagrad step {step}")
        # continue from the GPU's own state so the steps stay comparable
        wcur, Gcur = wg.copy(), (Gg.copy() if Gg is not None else Gcur)
        h.set_state(gu.cuda(wcur), gu.cuda(Gcur) if w.opt == "adagrad" else None)
    h.close()


@pytest.mark.parametrize("path", ["atomic", "sorted"])
@pytest.mark.parametrize("opt", ["sgd", "adagrad"])
def test_step_dyadic_bit_exact(opt, path):
    w = wl.make_workload("kaggle", B=1024, grad="dyadic", w0="dyadic")
    w.lr = 0.125
    h, o = gu.make_pair(w, opt=opt)
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS[path])
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    wg, Gg = h.get_state()
    w2, G2, _ = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B, w.grad_out,
                       opt, w.lr, w.eps)
    np.testing.assert_array_equal(gu.host(wg), w2)
    if opt == "adagrad":
        np.testing.assert_array_equal(gu.host(Gg), G2)
    h.close()


def test_dense_and_touched_updates_identical_on_both_paths():
    # Same exact gradient (dyadic inputs), two ways of visiting M and two
    # backward paths: same bits.
    w = wl.make_workload("tb", B=2048, grad="dyadic", w0="dyadic")
    res = []
    for mode, path in [(binding.UPDATE_DENSE, binding.PATH_ATOMIC),
                       (binding.UPDATE_TOUCHED, binding.PATH_ATOMIC),
                       (binding.UPDATE_DENSE, binding.PATH_SORTED),
                       (binding.UPDATE_TOUCHED, binding.PATH_SORTED)]:
        h, _ = gu.make_pair(w, opt="adagrad")
        h.set_option(binding.OPT_UPDATE_MODE, mode)
        h.set_option(binding.OPT_BACKWARD_PATH, path)
        for _ in range(2):
            h.forward(*_batch_cuda(w), w.B)
            h.backward_update(gu.cuda(w.grad_out), 0.01)
        wg, Gg = h.get_state()
        res.append((gu.host(wg), gu.host(Gg)))
        h.close()
    for r in res[1:]:
        np.testing.assert_array_equal(res[0][0], r[0])
        np.testing.assert_array_equal(res[0][1], r[1])


def test_sorted_path_reports_collision_rate():
    # rho = 1 - distinct blocks / (ids * chunks), from the global sort's
    # counters; the segment-local sort counts no distinct blocks (-1)
    t = gu.torch()
    w = wl.make_workload("tb", B=4096)
    h, o = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_SORT_SCOPE, binding.SORT_LOCAL)
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    t.cuda.synchronize()
    assert h.info()["last_collision_rate"] == -1.0
    h.set_option(binding.OPT_SORT_SCOPE, binding.SORT_GLOBAL)
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    t.cuda.synchronize()
    info = h.info()
    locs, _ = o.locations(w.indices, w.offsets, w.B)
    want = 1.0 - np.unique(locs).shape[0] / locs.shape[0]
    assert 0.0 < want < 1.0
    assert info["last_path"] == binding.PATH_SORTED
    assert abs(info["last_collision_rate"] - want) < 1e-12
    h.close()


@pytest.mark.parametrize("name,B", [("microbench", 10240), ("multihot", 4096), ("tb", 8192)])
def test_fp32_accumulation_within_recursive_sum_bound(name, B):
    # PSS_ACCUM_F32: the gradient is a recursive fp32 sum in atomic order, so
    # element e with n_e contributions may be off by (n_e - 1) u A_e (Higham).
    w = wl.make_workload(name, B=B)
    h, o = gu.make_pair(w)
    h.set_option(binding.OPT_ACCUM, binding.ACCUM_F32)
    h.forward(*_batch_cuda(w), w.B)
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    ref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    n = o.grad(w.indices, w.offsets, w.B, np.ones_like(w.grad_out))
    bound = np.maximum(n - 1, 1) * gu.U32 * A + gu.U32 * np.abs(ref)
    assert np.all(np.abs(g.astype(np.float64) - ref) <= bound)
    # SGD scattered straight into M: same bound on the step, plus the operand rounding
    h.forward(*_batch_cuda(w), w.B)
    if w.opt == "sgd":
        h.backward_update(gu.cuda(w.grad_out), w.lr)
        w2, _, _ = o.step(w.w0, None, w.indices, w.offsets, w.B, w.grad_out, "sgd", w.lr)
        err = np.abs(gu.host(h.get_weights()).astype(np.float64) - w2)
        scale = np.abs(w.w0).astype(np.float64) + w.lr * A
        assert np.all(err <= np.maximum(n, 1) * gu.U32 * scale + 2 * gu.U32 * np.abs(w2))
    h.close()


# --------------------------------------------------------------------------
# full sizes of the named workloads (default launch configuration)
@pytest.mark.parametrize("name", ["tiny", "kaggle", "tb", "multihot", "microbench"])
def test_full_size_step(name):
    w = wl.make_workload(name)
    h, o = gu.make_pair(w)
    idx, off = _batch_cuda(w)
    out = gu.host(h.forward(idx, off, w.B)).ravel()
    ref, bad = o.forward(w.w0, w.indices, w.offsets, w.B)
    assert bad == -1
    gu.check_forward(out, ref, _abs_pool(o, w.w0, w), what=f"{name} forward")
    del out, ref
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    wg, Gg = h.get_state()
    w2, G2, g32 = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B, w.grad_out,
                         w.opt, w.lr, w.eps)
    A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    if w.opt == "sgd":
        gu.check_sgd(gu.host(wg), w2, A, w.lr, what=f"{name} sgd")
    else:
        gu.check_adagrad(gu.host(wg), gu.host(Gg), w2, G2, g32, A, w.lr, what=f"{name} adagrad")
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()


# --------------------------------------------------------------------------
# scalar-column layouts with several columns per lane (VW = 1, KC = 2 or 4):
# d > 32 with d, Z or G not a multiple of 4 -- the paper's arbitrary offsets
# (G = 1) at the Criteo shapes, and the chunk-size study's small chunks
LAYOUT_CASES = [
    dict(name="tb", B=2048, G=1),                               # KC = 4, Adagrad
    dict(name="microbench", B=1024, Z=1, G=1),                  # HashedNet, J = 128
    dict(name="microbench", B=1024, Z=2, G=1),                  # J = 64
    dict(name="microbench", B=2048, Z=8),                       # J = 16, 32 ids per round
    dict(name="multihot", B=512, G=1, bag=("uniform", 0, 40)),  # KC = 2, ragged bags
]


@pytest.mark.parametrize("path", ["atomic", "sorted"])
@pytest.mark.parametrize("case", LAYOUT_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_scalar_layout_parity(case, path):
    w = _wl(case)
    h, o = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS[path])
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, bad = o.forward(w.w0, w.indices, w.offsets, w.B)
    assert bad == -1
    gu.check_forward(out, ref, _abs_pool(o, w.w0, w), what="scalar-layout forward")
    del out, ref
    grads = [("workload", w.grad_out)]
    if case["name"] == "microbench":
        # the paper's micro-benchmark loss (all ones) and a signed gradient
        grads.append(("normal", wl.make_batch(w.cards, w.B, w.d, case.get("bag", ("one",)),
                                              ("zipf", 1.05), seed=w.seed, batch=0)[2]))
    for gname, go in grads:
        h.forward(*_batch_cuda(w), w.B)
        g = gu.host(h.backward_grad(gu.cuda(go)))
        A = o.grad(w.indices, w.offsets, w.B, np.abs(go))
        gu.check_grad(g, o.grad(w.indices, w.offsets, w.B, go), A,
                      what=f"scalar-layout grad ({gname})")
        assert h.info()["last_path"] == PATHS[path]
    # three fused steps with fresh batches, state carried on both sides
    wcur, Gcur = w.w0.copy(), np.zeros(w.M, dtype=np.float32)
    h.set_state(gu.cuda(wcur), gu.cuda(Gcur) if w.opt == "adagrad" else None)
    cfg = wl.CONFIGS[case["name"]]
    for step in range(3):
        batch = (w.indices, w.offsets, w.grad_out) if step == 0 else wl.make_batch(
            w.cards, w.B, w.d, case.get("bag", cfg["bag"]), cfg["ids"], seed=w.seed, batch=step,
            grad=cfg.get("grad", "normal"))
        wg, Gg, w2, G2, g32, A = _run_step(w, h, o, wcur, Gcur, batch)
        if w.opt == "sgd":
            gu.check_sgd(wg, w2, A, w.lr, what=f"scalar-layout sgd step {step}")
        else:
            gu.check_adagrad(wg, Gg, w2, G2, g32, A, w.lr, what=f"scalar-layout adagrad step {step}")
        wcur, Gcur = w2, (G2 if w.opt == "adagrad" else Gcur)
        h.set_state(gu.cuda(wcur), gu.cuda(Gcur) if w.opt == "adagrad" else None)
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()


def _sub_batch(w, rows):
    """Bags of the given batch rows, all tables, as a smaller batch."""
    rows = np.asarray(rows)
    idx_parts, lens = [], []
    for t in range(w.T):
        for b in rows:
            s = t * w.B + b
            seg = w.indices[w.offsets[s]:w.offsets[s + 1]]
            idx_parts.append(seg)
            lens.append(seg.shape[0])
    off = np.zeros(len(lens) + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    return np.concatenate(idx_parts).astype(np.int64), off


SWEEP = ([(lm, "auto") for lm in (18, 20, 22, 24, 26, 28, 30, 32, 33)] +
         [(lm, "atomic") for lm in (28, 30, 32, 33)] +
         [(lm, "global") for lm in (24, 30)] +
         [(lm, "deterministic") for lm in (20, 26, 30)])


@pytest.mark.parametrize("logM,path", SWEEP, ids=[f"2^{lm}-{p}" for lm, p in SWEEP])
def test_compression_sweep(logM, path):
    """Criteo-TB shape with M from 2^18 to 2^33 fp32 (1 MB .. 32 GB).  Up to
    2^26 everything is compared; above, sampled rows and sampled elements
    (touched and untouched) are compared with the oracle evaluated one by one.
    AUTO takes the sorted path here (the segment-local sort; "global" sorts
    all pairs at once: counting sort at 2^24, radix sort at 2^30); the atomic
    path is forced at the large sizes too."""
    t = gu.torch()
    M = 1 << logM
    w = wl.make_workload("sweep", M=M)
    h, o = gu.make_pair(w)
    if path == "deterministic":
        h.set_option(binding.OPT_DETERMINISTIC, 1)
    if path == "global":
        h.set_option(binding.OPT_SORT_SCOPE, binding.SORT_GLOBAL)
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS.get(path, binding.PATH_AUTO))
    idx, off = _batch_cuda(w)
    out = h.forward(idx, off, w.B)
    rng = np.random.default_rng(logM)
    rows = np.sort(rng.choice(w.B, size=64, replace=False))
    sidx, soff = _sub_batch(w, rows)
    w0s = w.w0 if w.w0 is not None else None
    if w0s is not None:
        ref, _ = o.forward(w0s, sidx, soff, rows.shape[0])
        absr, _ = o.forward(np.abs(w0s), sidx, soff, rows.shape[0])
    else:
        # the oracle's pooling over a compact copy of the touched blocks: block
        # k of the copy holds the L elements at the k-th distinct location, and
        # the locations are remapped to k * L
        locs, _ = o.locations(sidx, soff, rows.shape[0])
        starts, inv = np.unique(locs, return_inverse=True)
        compact = w.w0_at((starts[:, None] + np.arange(o.L)[None, :]).ravel()).astype(np.float32)
        clocs = inv.reshape(-1).astype(np.int64) * o.L
        ref = o.pool(compact, clocs, soff, rows.shape[0], sidx.shape[0])
        absr = o.pool(np.abs(compact), clocs, soff, rows.shape[0], sidx.shape[0])
    got = gu.host(out[t.from_numpy(rows).cuda()]).ravel()
    gu.check_forward(got, ref, absr, what=f"sweep 2^{logM} forward")
    del out
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    if logM <= 26:
        wg, Gg = h.get_state()
        w2, G2, g32 = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B,
                             w.grad_out, w.opt, w.lr, w.eps)
        A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
        gu.check_adagrad(gu.host(wg), gu.host(Gg), w2, G2, g32, A, w.lr,
                         what=f"sweep 2^{logM}")
    else:
        locs, _ = o.locations(w.indices, w.offsets, w.B)
        pick = rng.choice(locs.shape[0], size=3000, replace=False)
        touched = (locs[pick][:, None] + np.arange(o.L)[None, :]).ravel()
        elems = np.unique(np.concatenate([touched, rng.integers(0, M, 20000)]))
        g_at = o.grad_at(w.indices, w.offsets, w.B, w.grad_out, elems)
        A_at = o.grad_at(w.indices, w.offsets, w.B, np.abs(w.grad_out), elems)
        w_s = w.w0_at(elems).astype(np.float32).copy()
        G_s = np.zeros(elems.shape[0], np.float32)
        g32 = g_at.astype(np.float32)
        o.adagrad(w_s, G_s, g32, w.lr, w.eps)
        wg, Gg = h.get_state()
        sel = t.from_numpy(elems).cuda()
        gu.check_adagrad(gu.host(wg[sel]), gu.host(Gg[sel]), w_s, G_s, g32, A_at, w.lr,
                         what=f"sweep 2^{logM} sampled")
        del wg, Gg
    assert h.info()["last_path"] == (binding.PATH_ATOMIC if path == "atomic" else
                                     binding.PATH_SORTED)
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()
    t.cuda.empty_cache()


# --------------------------------------------------------------------------
# the deterministic sorted path (stable radix sort), with automatic digits and
# with narrow ones: 4 or 7 bits per pass give two to six passes
DIGIT_CASES = [
    dict(name="tb", B=2048),                                  # 32-float chunks, staged reduce
    dict(name="multihot", B=256),                             # multi-id bags
    dict(name="multihot", B=301, bag=("uniform", 0, 6)),      # empty bags, ragged tail
    dict(name="tb", B=300, d=200, Z=32),                      # warp reduce, short last chunk
    dict(name="kaggle", Z=3, G=2, B=300),                     # lane-group reduce
    dict(name="tiny", Z=1, G=1),                              # one element per block
]


@pytest.mark.parametrize("bits", [0, 4, 7])
@pytest.mark.parametrize("signed", [False, True], ids=["unsigned", "signed"])
@pytest.mark.parametrize("case", DIGIT_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_sorted_digit_bits_parity(case, signed, bits):
    from oracle import OraclePSS
    w = _wl(case)
    h, o_u = gu.make_pair(w)
    o = o_u
    if signed:
        o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, signed=True)
        h.set_option(binding.OPT_SIGNED, 1)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    h.set_option(binding.OPT_SORT_DIGIT_BITS, bits)
    assert h.get_option(binding.OPT_SORT_DIGIT_BITS) == bits
    assert h.info()["R"] > (1 << bits)             # at least two passes when narrow
    idx, off = _batch_cuda(w)
    out = gu.host(h.forward(idx, off, w.B)).ravel()
    ref, _ = o.forward(w.w0, w.indices, w.offsets, w.B)
    gu.check_forward(out, ref, _abs_pool(o_u, w.w0, w), what="narrow-digit forward")
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    A = o_u.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, o.grad(w.indices, w.offsets, w.B, w.grad_out), A, what="narrow-digit grad")
    assert h.info()["last_path"] == binding.PATH_SORTED
    # a step with each update pass
    for mode in (binding.UPDATE_TOUCHED, binding.UPDATE_DENSE):
        h.set_state(gu.cuda(w.w0), gu.cuda(np.zeros(w.M, np.float32)) if w.opt == "adagrad" else None)
        h.set_option(binding.OPT_UPDATE_MODE, mode)
        wg, Gg, w2, G2, g32, _ = _run_step(w, h, o, w.w0, np.zeros(w.M, np.float32),
                                           (w.indices, w.offsets, w.grad_out))
        if w.opt == "sgd":
            gu.check_sgd(wg, w2, A, w.lr, what=f"narrow-digit sgd, update mode {mode}")
        else:
            gu.check_adagrad(wg, Gg, w2, G2, g32, A, w.lr,
                             what=f"narrow-digit adagrad, update mode {mode}")
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()


@pytest.mark.parametrize("opt", ["sgd", "adagrad"])
def test_sorted_narrow_digits_dyadic_bit_exact(opt):
    # dyadic inputs: every sum is exact, so a five-pass sort must still give
    # the oracle's bits
    w = wl.make_workload("kaggle", B=1024, grad="dyadic", w0="dyadic")
    w.lr = 0.125
    h, o = gu.make_pair(w, opt=opt)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    h.set_option(binding.OPT_SORT_DIGIT_BITS, 4)
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    wg, Gg = h.get_state()
    w2, G2, _ = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B, w.grad_out,
                       opt, w.lr, w.eps)
    np.testing.assert_array_equal(gu.host(wg), w2)
    if opt == "adagrad":
        np.testing.assert_array_equal(gu.host(Gg), G2)
    h.close()


def test_sort_digit_bits_option_rules():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    assert h.get_option(binding.OPT_SORT_DIGIT_BITS) == 0
    assert h.get_option(binding.OPT_DETERMINISTIC) == 0
    for bad in (2, -1):
        with pytest.raises(binding.PSSError):
            h.set_option(binding.OPT_DETERMINISTIC, bad)
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    assert h.get_option(binding.OPT_DETERMINISTIC) == 1
    for bad in (1, 3, 12, -1):
        with pytest.raises(binding.PSSError) as e:
            h.set_option(binding.OPT_SORT_DIGIT_BITS, bad)
        assert e.value.status == binding.PSS_ERR_INVALID_ARG
    h.forward(*_batch_cuda(w), w.B)
    h.set_option(binding.OPT_SORT_DIGIT_BITS, 4)     # the batch stays: nothing depends on it
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    h.set_option(binding.OPT_SORT_DIGIT_BITS, 11)
    assert h.get_option(binding.OPT_SORT_DIGIT_BITS) == 11
    h.close()


# --------------------------------------------------------------------------
# signed hashing (NEXT row: a +-1 per (id, chunk) from a second hash)
SIGNED_CASES = [
    dict(name="tiny"),
    dict(name="kaggle"),
    dict(name="tb", B=4096),
    dict(name="multihot", B=1024),
    dict(name="multihot", B=777, bag=("uniform", 0, 6)),      # empty bags, ragged tail
    dict(name="tiny", Z=1, G=1),                              # scalar kernels
    dict(name="kaggle", Z=3, G=2, B=300),                     # Z does not divide d
    dict(name="tb", B=500, d=200, Z=32),                      # two columns per lane
]


def _signed_pair(w, path):
    from oracle import OraclePSS
    h, o_u = gu.make_pair(w)
    o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, signed=True)
    h.set_option(binding.OPT_SIGNED, 1)
    _set_path(h, path)
    return h, o, o_u


@pytest.mark.parametrize("path", ["atomic", "sorted-global", "sorted-local"])
@pytest.mark.parametrize("case", SIGNED_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_signed_hashing_forward_and_grad_parity(case, path):
    w = _wl(case)
    h, o, o_u = _signed_pair(w, path)
    assert h.info()["signed_hash"] == 1
    assert (h.info()["A2"], h.info()["B2"]) == (o.A2, o.B2)
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, bad = o.forward(w.w0, w.indices, w.offsets, w.B)
    assert bad == -1
    # |s * w| = |w|: the unsigned oracle gives the conditioning bounds
    gu.check_forward(out, ref, _abs_pool(o_u, w.w0, w), what="signed forward")
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    gref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    A = o_u.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, gref, A, what="signed grad")
    assert h.info()["last_path"] == PATHS[path.split("-")[0]]
    h.close()


@pytest.mark.parametrize("path", ["atomic", "sorted"])
@pytest.mark.parametrize("opt", ["sgd", "adagrad"])
def test_signed_hashing_step_dyadic_bit_exact(opt, path):
    # dyadic inputs: every sum is exact, so the signed step must give the
    # oracle's bits on both paths
    w = wl.make_workload("kaggle", B=1024, grad="dyadic", w0="dyadic", opt=opt)
    w.lr = 0.125
    h, o, _ = _signed_pair(w, path)
    h.forward(*_batch_cuda(w), w.B)
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, _ = o.forward(w.w0, w.indices, w.offsets, w.B)
    np.testing.assert_array_equal(out, ref)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    wg, Gg = h.get_state()
    w2, G2, _ = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B, w.grad_out,
                       opt, w.lr, w.eps)
    np.testing.assert_array_equal(gu.host(wg), w2)
    if opt == "adagrad":
        np.testing.assert_array_equal(gu.host(Gg), G2)
    h.close()


def test_signed_option_forgets_the_batch_and_needs_small_R():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    h.forward(*_batch_cuda(w), w.B)
    h.set_option(binding.OPT_SIGNED, 1)
    with pytest.raises(binding.PSSError) as e:
        h.backward_update(gu.cuda(w.grad_out), w.lr)
    assert e.value.status == binding.PSS_ERR_STATE
    assert h.get_option(binding.OPT_SIGNED) == 1
    with pytest.raises(binding.PSSError):
        h.set_option(binding.OPT_SIGNED, 2)
    h.close()
    # R >= 2^31 block starts: the sign cannot travel in bit 31
    big = binding.PSS(w.cards, dim=16, M=(1 << 31) + 64, Z=16, G=1, seed=0, optimizer="sgd")
    with pytest.raises(binding.PSSError) as e:
        big.set_option(binding.OPT_SIGNED, 1)
    assert e.value.status == binding.PSS_ERR_UNSUPPORTED
    big.close()


# --------------------------------------------------------------------------
# circular array (NEXT row: R = M/G starts, blocks past M wrap to its start)
CIRC_CASES = [
    dict(name="tiny", M=256),                 # 64 starts, 3 of them wrap
    dict(name="tiny"),
    dict(name="kaggle"),
    dict(name="tb", B=4096),
    dict(name="multihot", B=1024),
    dict(name="tiny", Z=1, G=1, M=999),       # scalar kernels
    dict(name="kaggle", Z=3, G=2, B=300),     # Z does not divide d
]


def _circ_pair(w, path, signed=False):
    from oracle import OraclePSS
    h, _ = gu.make_pair(w)
    o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, signed=signed, circular=True)
    o_abs = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, circular=True)
    h.set_option(binding.OPT_CIRCULAR, 1)
    if signed:
        h.set_option(binding.OPT_SIGNED, 1)
    _set_path(h, path)
    h.set_weights(gu.cuda(w.w0))      # (re)load: refreshes the mirror of M[0 .. L)
    return h, o, o_abs


@pytest.mark.parametrize("signed", [False, True])
@pytest.mark.parametrize("path", ["atomic", "sorted-global", "sorted-local"])
@pytest.mark.parametrize("case", CIRC_CASES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_circular_forward_and_grad_parity(case, path, signed):
    w = _wl(case)
    h, o, o_abs = _circ_pair(w, path, signed)
    info = h.info()
    assert info["circular"] == 1 and info["R"] == o.R == w.M // w.G
    np.testing.assert_array_equal(gu.host(h.compute_locations(*_batch_cuda(w), w.B)),
                                  o.locations(w.indices, w.offsets, w.B)[0])
    out = gu.host(h.forward(*_batch_cuda(w), w.B)).ravel()
    ref, bad = o.forward(w.w0, w.indices, w.offsets, w.B)
    assert bad == -1
    gu.check_forward(out, ref, _abs_pool(o_abs, w.w0, w), what="circular forward")
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    gref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    A = o_abs.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, gref, A, what="circular grad")
    h.close()


@pytest.mark.parametrize("signed", [False, True], ids=["unsigned", "signed"])
@pytest.mark.parametrize("case", [dict(name="tb", B=2048), dict(name="kaggle", Z=3, G=2, B=300)],
                         ids=["tb", "kaggle-Z3-G2"])
def test_circular_with_narrow_digits(case, signed):
    # circular array and a many-pass radix sort: the wrapped blocks'
    # contributions fold into the head after the sorted reduce
    w = _wl(case)
    h, o, o_abs = _circ_pair(w, "sorted", signed)
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    h.set_option(binding.OPT_SORT_DIGIT_BITS, 5)
    h.forward(*_batch_cuda(w), w.B)
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    A = o_abs.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, o.grad(w.indices, w.offsets, w.B, w.grad_out), A, what="circular narrow-digit grad")
    assert h.info()["last_path"] == binding.PATH_SORTED
    h.close()


@pytest.mark.parametrize("path", ["atomic", "sorted"])
@pytest.mark.parametrize("opt", ["sgd", "adagrad"])
def test_circular_steps_dyadic_bit_exact(opt, path):
    # three steps: each forward reads the wrapped blocks through the mirror the
    # previous update refreshed; dyadic inputs make every result exact
    w = wl.make_workload("tiny", M=256, grad="dyadic", w0="dyadic", opt=opt)
    w.lr = 0.125
    h, o, _ = _circ_pair(w, path)
    wcur, Gcur = w.w0.copy(), np.zeros(w.M, np.float32)
    for k in range(3):
        wk = wl.make_workload("tiny", M=256, grad="dyadic", w0="dyadic", opt=opt, batch=k)
        out = gu.host(h.forward(*_batch_cuda(wk), wk.B)).ravel()
        ref, _ = o.forward(wcur, wk.indices, wk.offsets, wk.B)
        np.testing.assert_array_equal(out, ref)
        h.backward_update(gu.cuda(wk.grad_out), w.lr)
        wcur, Gcur, _ = o.step(wcur, Gcur, wk.indices, wk.offsets, wk.B, wk.grad_out, opt, w.lr,
                               w.eps)
        wg, Gg = h.get_state()
        np.testing.assert_array_equal(gu.host(wg), wcur)
        if opt == "adagrad":
            np.testing.assert_array_equal(gu.host(Gg), Gcur)
    h.close()


def test_circular_option_rules():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    R0 = h.info()["R"]
    h.forward(*_batch_cuda(w), w.B)
    h.set_option(binding.OPT_CIRCULAR, 1)
    assert h.info()["R"] == w.M // w.G != R0
    with pytest.raises(binding.PSSError) as e:
        h.backward_update(gu.cuda(w.grad_out), w.lr)
    assert e.value.status == binding.PSS_ERR_STATE
    h.set_option(binding.OPT_CIRCULAR, 0)
    assert h.info()["R"] == R0 and h.get_option(binding.OPT_CIRCULAR) == 0
    h.close()
    odd = binding.PSS(w.cards, dim=16, M=1002, Z=16, G=4, seed=0, optimizer="sgd")
    with pytest.raises(binding.PSSError) as e:
        odd.set_option(binding.OPT_CIRCULAR, 1)
    assert e.value.status == binding.PSS_ERR_UNSUPPORTED
    odd.close()


# --------------------------------------------------------------------------
# host buffers through the same C-ABI calls (the end-to-end path)
# Criteo-TB batch 8192: 109 MB of pooled output, which the forward computes in
# chunks of batch rows and downloads chunk by chunk into pinned host memory
@pytest.mark.parametrize("name,B", [("kaggle", None), ("tb", 8192)])
def test_host_buffers_match_device_buffers(name, B):
    # dyadic inputs: every sum is exact, so both paths must give the same bits
    t = gu.torch()
    w = wl.make_workload(name, B=B, grad="dyadic", w0="dyadic")
    w.lr = 0.125
    h1, _ = gu.make_pair(w, opt="sgd")
    h2, _ = gu.make_pair(w, opt="sgd")
    out_d = gu.host(h1.forward(*_batch_cuda(w), w.B))
    idx_h = t.from_numpy(w.indices).pin_memory()
    off_h = t.from_numpy(w.offsets).pin_memory()
    out_h = h2.forward(idx_h, off_h, w.B)
    t.cuda.synchronize()
    assert not out_h.is_cuda
    np.testing.assert_array_equal(out_h.numpy(), out_d)
    # pageable host memory works too
    out_p = t.empty(out_h.shape, dtype=t.float32)
    h2.forward(t.from_numpy(w.indices), t.from_numpy(w.offsets), w.B, out=out_p)
    t.cuda.synchronize()
    np.testing.assert_array_equal(out_p.numpy(), out_d)
    h1.backward_update(gu.cuda(w.grad_out), w.lr)
    h2.backward_update(t.from_numpy(w.grad_out).pin_memory(), w.lr)
    np.testing.assert_array_equal(gu.host(h2.get_weights()), gu.host(h1.get_weights()))
    h1.close()
    h2.close()


@pytest.mark.parametrize("path", ["sorted", "atomic", "atomic-f32"])
def test_host_gradient_upload_is_ordered(path):
    # A host upstream gradient is copied in on the library's own copy stream
    # (overlapping the forward and the output download).  Three steps through
    # host buffers, with the pinned gradient buffer overwritten right after
    # each step's stream synchronisation, must match device buffers bit for
    # bit (dyadic inputs: every sum is exact on every path).
    t = gu.torch()
    w = wl.make_workload("kaggle", grad="dyadic", w0="dyadic")
    w.lr = 0.125
    h1, _ = gu.make_pair(w, opt="sgd")
    h2, _ = gu.make_pair(w, opt="sgd")
    for h in (h1, h2):
        h.set_option(binding.OPT_BACKWARD_PATH,
                     binding.PATH_SORTED if path == "sorted" else binding.PATH_ATOMIC)
        if path == "atomic-f32":
            h.set_option(binding.OPT_ACCUM, binding.ACCUM_F32)
    g_host = t.empty(w.grad_out.shape, dtype=t.float32).pin_memory()
    out_h = t.empty((w.B, w.T, w.d), dtype=t.float32).pin_memory()
    for k in range(3):
        wk = wl.make_workload("kaggle", grad="dyadic", w0="dyadic", batch=k)
        h1.forward(*_batch_cuda(wk), wk.B)
        h1.backward_update(gu.cuda(wk.grad_out), w.lr)
        h2.forward(t.from_numpy(wk.indices).pin_memory(), t.from_numpy(wk.offsets).pin_memory(),
                   wk.B, out=out_h)
        g_host.copy_(t.from_numpy(wk.grad_out))
        h2.backward_update(g_host, w.lr)
        t.cuda.synchronize()
        g_host.fill_(float("nan"))
    np.testing.assert_array_equal(gu.host(h2.get_weights()), gu.host(h1.get_weights()))
    # a batch whose bags are all empty, with a host gradient: nothing changes
    before = gu.host(h2.get_weights())
    empty_off = np.zeros(w.T * w.B + 1, dtype=np.int64)
    h2.forward(t.from_numpy(np.zeros(0, dtype=np.int64)), t.from_numpy(empty_off), w.B, out=out_h)
    g_host.copy_(t.from_numpy(w.grad_out))
    h2.backward_update(g_host, w.lr)
    t.cuda.synchronize()
    np.testing.assert_array_equal(gu.host(h2.get_weights()), before)
    h1.close()
    h2.close()


# --------------------------------------------------------------------------
# errors: reported, never a trap
@pytest.mark.parametrize("path", ["atomic", "sorted"])
def test_out_of_range_ids_are_skipped_and_reported(path):
    w = wl.make_workload("tiny")
    idx = w.indices.copy()
    idx[100] = 5000          # beyond the 1000-id table
    idx[37] = -3
    h, o = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, PATHS[path])
    out = gu.host(h.forward(gu.cuda(idx), gu.cuda(w.offsets), w.B)).ravel()
    st, first = h.get_error()
    assert st == binding.PSS_ERR_INDEX_RANGE and first == 37
    ref, bad = o.forward(w.w0, idx, w.offsets, w.B)
    assert bad == 37
    np.testing.assert_array_equal(out, ref)
    assert h.get_error() == (binding.PSS_OK, -1)     # cleared by the read
    # the backward skips the same ids
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    gref = o.grad(idx, w.offsets, w.B, w.grad_out)
    A = o.grad(idx, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, gref, A)
    h.close()


@pytest.mark.parametrize("path", ["sorted-local", "sorted-global"])
def test_out_of_range_ids_in_local_segments(path):
    # 32-float chunks (the segment-local sort): bad ids scattered over several
    # 8192-pair segments, one segment with many; each segment's valid entries
    # are counted and the rest of its range is never read
    w = wl.make_workload("tb", B=3001)
    idx = w.indices.copy()
    rng = np.random.default_rng(5)
    bad = np.concatenate([rng.choice(idx.shape[0], 40, replace=False),
                          np.arange(5000, 5600)])
    idx[bad] = -1
    idx[bad[:20]] = 1 << 40
    h, o = gu.make_pair(w)
    _set_path(h, path)
    h.forward(gu.cuda(idx), gu.cuda(w.offsets), w.B)
    st, first = h.get_error()
    assert st == binding.PSS_ERR_INDEX_RANGE and first == int(bad.min())
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    gref = o.grad(idx, w.offsets, w.B, w.grad_out)
    A = o.grad(idx, w.offsets, w.B, np.abs(w.grad_out))
    gu.check_grad(g, gref, A)
    h.close()


@pytest.mark.parametrize("name,B", [("tb", 3001), ("multihot", 777)])
@pytest.mark.parametrize("opt", ["sgd", "adagrad"])
def test_local_sort_step_dyadic_bit_exact(name, B, opt):
    # dyadic inputs: every partial sum is exact, so the segment-local
    # grouping gives the oracle's bits whatever the order of its additions
    w = wl.make_workload(name, B=B, grad="dyadic", w0="dyadic")
    w.lr = 0.125
    h, o = gu.make_pair(w, opt=opt)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_SORT_SCOPE, binding.SORT_LOCAL)
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    wg, Gg = h.get_state()
    w2, G2, _ = o.step(w.w0, np.zeros(w.M, np.float32), w.indices, w.offsets, w.B, w.grad_out,
                       opt, w.lr, w.eps)
    np.testing.assert_array_equal(gu.host(wg), w2)
    if opt == "adagrad":
        np.testing.assert_array_equal(gu.host(Gg), G2)
    assert h.info()["last_collision_rate"] == -1.0     # the local sort ran
    h.close()


@pytest.mark.parametrize("name,B,M,want", [("kaggle", 2048, None, "dense"), ("tb", 64, None, "dense"),
                                            ("sweep", 1024, 1 << 25, "touched"),
                                            ("sweep", 65536, 1 << 25, "dense")])
def test_update_mode_auto_rule(name, B, M, want):
    # AUTO: dense while 16 * M bytes fit in half the L2 or M <= pairs * L;
    # the touched pass otherwise (pss_info.last_update says which ran)
    t = gu.torch()
    w = wl.make_workload(name, B=B, M=M)
    h, _ = gu.make_pair(w)
    h.forward(*_batch_cuda(w), w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    t.cuda.synchronize()
    l2 = t.cuda.get_device_properties(0).L2_cache_size
    pairs_l = w.indices.shape[0] * (-(-w.d // w.Z)) * min(w.Z, w.d)
    assert (want == "touched") == (16 * w.M > l2 // 2 and w.M > pairs_l)
    assert h.info()["last_update"] == {"dense": binding.UPDATE_DENSE,
                                       "touched": binding.UPDATE_TOUCHED}[want]
    assert h.get_error() == (binding.PSS_OK, -1)
    h.close()


def test_sort_scope_option_rules():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    assert h.get_option(binding.OPT_SORT_SCOPE) == binding.SORT_AUTO
    for bad in (-1, 3):
        with pytest.raises(binding.PSSError):
            h.set_option(binding.OPT_SORT_SCOPE, bad)
    for v in (binding.SORT_GLOBAL, binding.SORT_LOCAL, binding.SORT_AUTO):
        h.set_option(binding.OPT_SORT_SCOPE, v)
        assert h.get_option(binding.OPT_SORT_SCOPE) == v
    h.close()


@pytest.mark.parametrize("name,B,local", [("tb", 1024, True), ("tb", 65536, False),
                                          ("microbench", 10240, True), ("tiny", 256, False)])
def test_sort_scope_auto_rule(name, B, local):
    # AUTO: local where the chunks tile the rows and the batch has at most
    # 3 pairs per block start (R > 2^22 aside); the collision rate tells
    # which ran (-1 after a local pass)
    t = gu.torch()
    w = wl.make_workload(name, B=B)
    h, _ = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    idx, off = _batch_cuda(w)
    go = gu.cuda(w.grad_out)
    for _ in range(2):        # the global sort's counts reach the host by the next call
        h.forward(idx, off, w.B)
        h.backward_update(go, w.lr)
    t.cuda.synchronize()
    h.forward(idx, off, w.B)
    h.backward_update(go, w.lr)
    pairs = w.indices.shape[0] * (-(-w.d // w.Z))
    assert (pairs <= 3 * h.info()["R"]) == local or name == "tiny"
    assert (h.info()["last_collision_rate"] == -1.0) == local
    h.close()


def test_malformed_offsets_reported():
    w = wl.make_workload("tiny")
    off = w.offsets.copy()
    off[10] = off[11] + 5    # decreasing
    h, _ = gu.make_pair(w)
    h.forward(gu.cuda(w.indices), gu.cuda(off), w.B)
    st, first = h.get_error()
    assert st == binding.PSS_ERR_INDEX_RANGE and first == -2
    h.close()


def test_call_order_and_argument_errors():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    with pytest.raises(binding.PSSError) as e:
        h.backward_update(gu.cuda(w.grad_out), 0.1)
    assert e.value.status == binding.PSS_ERR_STATE
    with pytest.raises(binding.PSSError) as e:
        h.set_weights(gu.cuda(np.zeros(10, np.float32)))
    assert e.value.status == binding.PSS_ERR_INVALID_ARG
    with pytest.raises(binding.PSSError):
        h.set_option(99, 0)
    with pytest.raises(binding.PSSError):
        h.set_option(binding.OPT_BACKWARD_PATH, 7)
    h.close()


def test_empty_batch():
    w = wl.make_workload("tiny")
    h, _ = gu.make_pair(w)
    t = gu.torch()
    out = h.forward(t.zeros(0, dtype=t.int64, device="cuda"),
                    t.zeros(1, dtype=t.int64, device="cuda"), 0)
    assert out.numel() == 0
    h.backward_update(t.zeros(0, dtype=t.float32, device="cuda"), 0.1)
    wg = gu.host(h.get_weights())
    np.testing.assert_array_equal(wg, w.w0)
    # bags that are all empty: zero rows, no update
    off = np.zeros(w.T * 4 + 1, np.int64)
    out = gu.host(h.forward(t.zeros(0, dtype=t.int64, device="cuda"), gu.cuda(off), 4))
    assert out.shape == (4, w.T, w.d) and not out.any()
    h.close()


def test_profile_and_launch_counts():
    w = wl.make_workload("kaggle")
    h, _ = gu.make_pair(w)
    h.set_option(binding.OPT_PROFILE, 1)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_ATOMIC)
    h.set_option(binding.OPT_UPDATE_MODE, binding.UPDATE_DENSE)
    idx, off = _batch_cuda(w)
    go = gu.cuda(w.grad_out)
    before = h.info()["kernel_launches"]
    for _ in range(3):
        h.forward(idx, off, w.B)
        h.backward_update(go, w.lr)
    n_f, ms_f = h.profile(binding.K_FORWARD)
    n_s, ms_s = h.profile(binding.K_SCATTER)
    assert n_f == 3 and n_s == 3 and ms_f > 0 and ms_s > 0
    assert h.info()["kernel_launches"] - before == 9     # forward, scatter, update
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.reset_profile()
    before = h.info()["kernel_launches"]
    h.forward(idx, off, w.B)
    h.backward_update(go, w.lr)
    assert h.profile(binding.K_SORT)[0] == 1 and h.profile(binding.K_REDUCE)[0] == 1
    # forward, bucket count, 2 scan kernels, slot scatter, reduce, update
    assert h.info()["R"] < (1 << 22)
    assert h.info()["kernel_launches"] - before == 7
    # deterministic: forward, two radix passes of three kernels each (R < 2^22), reduce, update
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    before = h.info()["kernel_launches"]
    h.forward(idx, off, w.B)
    h.backward_update(go, w.lr)
    assert h.info()["kernel_launches"] - before == 9
    h.close()
    # 32-float chunks: forward, segment-local sort, reduce, update
    w = wl.make_workload("tb", B=2048)
    h, _ = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_SORT_SCOPE, binding.SORT_LOCAL)
    h.set_option(binding.OPT_UPDATE_MODE, binding.UPDATE_DENSE)
    idx, off = _batch_cuda(w)
    h.forward(idx, off, w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    before = h.info()["kernel_launches"]
    h.forward(idx, off, w.B)
    h.backward_update(gu.cuda(w.grad_out), w.lr)
    assert h.info()["kernel_launches"] - before == 4
    h.close()


def test_l2_probe_runs_and_rejects_bad_arguments():
    # the measurement hook behind bench.py's L2 peaks: every kind runs on a
    # device buffer; host buffers, bad kinds and unaligned sizes are refused
    t = gu.torch()
    buf = t.zeros(1 << 20, dtype=t.float32, device="cuda")
    for kind in (0, 1, 2, 3):
        binding.probe_l2(kind, buf, 16, 8)
    t.cuda.synchronize()
    for bad in (dict(kind=4, buf=buf), dict(kind=0, buf=t.zeros(1 << 20))):
        with pytest.raises(binding.PSSError) as e:
            binding.probe_l2(bad["kind"], bad["buf"], 16, 8)
        assert e.value.status == binding.PSS_ERR_INVALID_ARG


@pytest.mark.parametrize("name,B,want", [("tb", 1024, "atomic"), ("tb", 2048, "sorted"),
                                          ("kaggle", 8192, "atomic"),
                                          ("kaggle", 32768, "sorted")])
def test_auto_path_threshold(name, B, want):
    # AUTO picks the sorted path from 5M element adds (nnz * J * L) with
    # 32-element blocks and from 10M with shorter ones: the Criteo-TB shape
    # adds 3.4M at batch 1024 and 6.8M at 2048, the Criteo-Kaggle shape
    # (16-element blocks) 3.4M at batch 8192 and 13.6M at 32768
    w = wl.make_workload(name, B=B)
    h, o = gu.make_pair(w)
    assert h.get_option(binding.OPT_BACKWARD_PATH) == binding.PATH_AUTO
    h.forward(*_batch_cuda(w), w.B)
    g = gu.host(h.backward_grad(gu.cuda(w.grad_out)))
    assert h.info()["last_path"] == PATHS[want]
    gu.check_grad(g, o.grad(w.indices, w.offsets, w.B, w.grad_out),
                  o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out)))
    h.close()
