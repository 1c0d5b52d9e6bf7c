"""Determinism of the sorted backward path (Algorithm 1's sparse branch) with
PSS_OPT_DETERMINISTIC.

That mode orders every bucket's contributions by a stable radix sort (pair
order inside a bucket) and sums each run in that order, so two runs on
the same inputs give the same bits, and a training run can be stopped after
any step, checkpointed with pss_get_state, restored into a new handle with
pss_set_state, and continued to the same bits as an uninterrupted run.  The
inputs are the Criteo-TB shape at full batch with N(0,1) upstream gradients
(not dyadic: sums round, so only a fixed summation order gives equal bits).
"""
import numpy as np
import pytest

from paper_2207_10731_gb300 import binding, workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


def _bits(a):
    return np.ascontiguousarray(a).view(np.uint32)


def _batches(w, n):
    cfg = wl.CONFIGS[w.name]
    out = [(w.indices, w.offsets, w.grad_out)]
    for k in range(1, n):
        out.append(wl.make_batch(w.cards, w.B, w.d, cfg["bag"], cfg["ids"], seed=w.seed, batch=k,
                                 grad=cfg.get("grad", "normal")))
    return [(gu.cuda(i), gu.cuda(o), gu.cuda(g)) for i, o, g in out]


def _handle(w, state=None):
    h, _ = gu.make_pair(w)
    h.set_option(binding.OPT_BACKWARD_PATH, binding.PATH_SORTED)
    h.set_option(binding.OPT_DETERMINISTIC, 1)
    if state is not None:
        wv, Gv = state
        h.set_state(gu.cuda(wv), gu.cuda(Gv) if Gv is not None else None)
    return h


def _steps(h, w, batches):
    for idx, off, go in batches:
        h.forward(idx, off, w.B)
        h.backward_update(go, w.lr)
    wg, Gg = h.get_state()
    return gu.host(wg), (gu.host(Gg) if Gg is not None else None)


@pytest.mark.parametrize("name,B", [("tb", None), ("multihot", 4096)])
def test_sorted_path_two_runs_same_bits(name, B):
    w = wl.make_workload(name, B=B)
    batches = _batches(w, 2)
    runs = []
    for _ in range(2):
        h = _handle(w)
        runs.append(_steps(h, w, batches))
        assert h.info()["last_path"] == binding.PATH_SORTED
        h.close()
    np.testing.assert_array_equal(_bits(runs[0][0]), _bits(runs[1][0]))
    if runs[0][1] is not None:
        np.testing.assert_array_equal(_bits(runs[0][1]), _bits(runs[1][1]))
    # the gradient alone, twice on one handle
    h = _handle(w)
    idx, off, go = batches[0]
    h.forward(idx, off, w.B)
    g1 = gu.host(h.backward_grad(go))
    g2 = gu.host(h.backward_grad(go))
    np.testing.assert_array_equal(_bits(g1), _bits(g2))
    h.close()


def test_sorted_path_checkpoint_resume_same_bits():
    # 4 Adagrad steps straight through, against 2 steps, a checkpoint to host
    # memory, a new handle restored from it, and 2 more steps
    w = wl.make_workload("tb", B=16384)
    batches = _batches(w, 4)
    h = _handle(w)
    full = _steps(h, w, batches)
    h.close()
    h = _handle(w)
    ckpt = _steps(h, w, batches[:2])
    h.close()
    h = _handle(w, state=(ckpt[0].copy(), ckpt[1].copy()))
    resumed = _steps(h, w, batches[2:])
    h.close()
    np.testing.assert_array_equal(_bits(full[0]), _bits(resumed[0]))
    np.testing.assert_array_equal(_bits(full[1]), _bits(resumed[1]))
