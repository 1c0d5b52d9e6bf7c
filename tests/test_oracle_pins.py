"""Pins for the CPU oracle: checks against things other than the oracle itself.

* published splitmix64 outputs (the seed -> hash-parameter generator);
* Python big-integer evaluation of the universal hash (Sec. 2.5);
* the explicit 0/1 mapping matrix P on tiny inputs: pooled forward = P w and
  gradient = P^T grad_out (Sec. 2.4 forward/backward), built with scipy.sparse
  from big-integer locations;
* the two branches of Algorithm 1 (dense scatter_add vs unique + scatter_add);
* special cases: an injective mapping is a plain embedding table (Def. 1,
  M = E) and must equal torch's embedding_bag(sum); the hashing trick (Sec. 2.5)
  is the case G = Z = d;
* invariants: all-ones upstream gradient gives integer contribution counts;
  total gradient mass equals sum over bags of |bag| * sum(grad_out row);
* optimizer steps against torch.optim.SGD / torch.optim.Adagrad and closed forms.
"""
import os

import numpy as np
import pytest
import scipy.sparse as sp

import oracle
from oracle import OraclePSS, OracleError
from paper_2207_10731_gb300 import workloads as wl
from tests import bigint_hash as bh

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_hex(name):
    vals = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                vals.append(int(line, 16))
    return vals


def test_splitmix64_published_sequence():
    want = _golden_hex("splitmix64_seed0.txt")
    got = [int(x) for x in oracle.splitmix64_seq(0, len(want))]
    assert got == want


def test_bigint_helper_matches_published_sequence():
    # the test-side helper derives (A, B0) from the same published stream
    s = _golden_hex("splitmix64_seed0.txt")
    A, B0 = bh.params(0)
    assert A == 1 + s[0] % (bh.P61 - 1)
    assert B0 == s[1] % bh.P61


@pytest.mark.parametrize("seed", [0, 1, 12345, 2**63 + 7])
def test_hash_params_from_seed(seed):
    assert oracle.hash_params(seed) == bh.params(seed)
    A, B0 = oracle.hash_params(seed)
    assert 1 <= A < bh.P61 and 0 <= B0 < bh.P61


@pytest.mark.parametrize("M,Z,G,d,T", [(16384, 16, 4, 16, 8), (2_500_000, 32, 4, 128, 26),
                                       (1 << 33, 32, 4, 128, 26), (1000, 1, 1, 7, 3),
                                       (257, 32, 1, 16, 2), (3 << 32, 32, 32, 64, 26)])
def test_locations_match_bigint(M, Z, G, d, T):
    rng = np.random.default_rng(1)
    cards = rng.integers(3, 40_000_000, size=T)
    o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=7)
    A, B0 = bh.params(7)
    L = min(Z, d)
    J = -(-d // Z)
    R = (M - L) // G + 1
    assert (o.A, o.B0, o.J, o.L, o.R) == (A, B0, J, L, R)
    for _ in range(400):
        t = int(rng.integers(0, T))
        i = int(rng.integers(0, cards[t]))
        j = int(rng.integers(0, J))
        want = bh.location(A, B0, R, G, T, J, i, t, j)
        got = o.location(i, t, j)
        assert got == want
        assert 0 <= got <= M - L and got % G == 0
    # extreme ids
    for t in (0, T - 1):
        for i in (0, int(cards[t]) - 1):
            for j in (0, J - 1):
                assert o.location(i, t, j) == bh.location(A, B0, R, G, T, J, i, t, j)


def test_bucket_uniformity_chi2():
    # 2-universal hash of distinct keys: bucket counts close to uniform.
    from scipy.stats import chi2
    o = OraclePSS([1 << 20], d=4, M=4 * 1000 + 0, Z=4, G=4, seed=3)
    assert o.R == 1000
    idx = np.arange(200_000, dtype=np.int64) * 5 + 11
    offs = np.arange(idx.shape[0] + 1, dtype=np.int64)
    locs, bad = o.locations(idx, offs, idx.shape[0])
    assert bad == -1
    counts = np.bincount(locs // 4, minlength=o.R)
    exp = idx.shape[0] / o.R
    stat = ((counts - exp) ** 2 / exp).sum()
    assert chi2.sf(stat, o.R - 1) > 1e-4


def _tiny_case(seed, T=2, B=4, d=16, M=256, Z=4, G=4, max_bag=3, dy=True):
    rng = np.random.default_rng(seed)
    cards = rng.integers(3, 50, size=T)
    lengths = rng.integers(0, max_bag + 1, size=T * B)
    offsets = np.zeros(T * B + 1, dtype=np.int64)
    np.cumsum(lengths, out=offsets[1:])
    idx = np.concatenate([rng.integers(0, cards[t], size=int(lengths[t * B:(t + 1) * B].sum()))
                          for t in range(T)]).astype(np.int64)
    if dy:
        w = wl.dyadic(rng, M)
        go = wl.dyadic(rng, B * T * d)
    else:
        w = rng.standard_normal(M).astype(np.float32)
        go = rng.standard_normal(B * T * d).astype(np.float32)
    return cards, idx, offsets, w, go


def _bruteforce_P(cards, idx, offsets, B, d, M, Z, G, seed):
    """Explicit 0/1 mapping matrix, rows (b, t, k) of the pooled output,
    columns = elements of the shared array; locations from big integers."""
    T = len(cards)
    A, B0 = bh.params(seed)
    L, J = min(Z, d), -(-d // Z)
    R = (M - L) // G + 1
    rows, cols = [], []
    for t in range(T):
        for b in range(B):
            s = t * B + b
            for q in range(offsets[s], offsets[s + 1]):
                i = int(idx[q])
                for k in range(d):
                    j, z = divmod(k, Z)
                    rows.append((b * T + t) * d + k)
                    cols.append(bh.location(A, B0, R, G, T, J, i, t, j) + z)
    data = np.ones(len(rows))
    return sp.coo_matrix((data, (rows, cols)), shape=(B * T * d, M)).tocsr()


@pytest.mark.parametrize("Z,G,d", [(1, 1, 16), (4, 4, 16), (16, 4, 16), (32, 4, 16),
                                   (32, 1, 16), (16, 1, 16), (4, 1, 10), (3, 2, 10),
                                   (32, 32, 16)])
def test_forward_and_grad_equal_bruteforce_matrix(Z, G, d):
    T, B, M = 2, 4, 256
    for seed in range(3):
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed)
        P = _bruteforce_P(cards, idx, off, B, d, M, Z, G, seed)
        out, bad = o.forward(w, idx, off, B)
        assert bad == -1
        # dyadic inputs: every partial sum is exact, so bits must agree
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
        g = o.grad(idx, off, B, go)
        np.testing.assert_array_equal(g, P.T @ go.astype(np.float64))


# --------------------------------------------------------------------------
# signed hashing: every (id, chunk) also carries a sign s = +-1 from a second
# hash of the same family (Sec. 2.5: the sketch comes from +-1 projections)
@pytest.mark.parametrize("seed", [0, 7, 2**63 + 7])
def test_sign_hash_matches_bigint(seed):
    cards = [1000, 37, 40_000_000]
    o = OraclePSS(cards, d=128, M=2_500_000, Z=32, G=4, seed=seed, signed=True)
    A2, B2 = bh.sign_params(seed)
    assert (o.A2, o.B2) == (A2, B2)
    assert (o.A, o.B0) != (o.A2, o.B2)
    rng = np.random.default_rng(seed % 1000)
    for _ in range(300):
        t = int(rng.integers(0, 3))
        i = int(rng.integers(0, cards[t]))
        j = int(rng.integers(0, o.J))
        assert o.sign(i, t, j) == bh.sign(A2, B2, 3, o.J, i, t, j)
    # unsigned instance: every sign is +1
    u = OraclePSS(cards, d=128, M=2_500_000, Z=32, G=4, seed=seed)
    assert all(u.sign(i, 0, 0) == 1 for i in range(50))


def test_signs_are_balanced():
    o = OraclePSS([10_000_000] * 4, d=128, M=2_500_000, Z=32, G=4, seed=3, signed=True)
    s = np.array([o.sign(i, t, j) for i in range(0, 4000, 3) for t in range(4) for j in range(4)])
    n = s.shape[0]
    # a fair coin: the count of -1 within 5 standard deviations of n/2
    assert abs((s == -1).sum() - n / 2) < 5 * np.sqrt(n / 4)


@pytest.mark.parametrize("Z,G,d", [(1, 1, 16), (4, 4, 16), (32, 4, 16), (3, 2, 10)])
def test_signed_forward_and_grad_equal_signed_bruteforce_matrix(Z, G, d):
    # the explicit +-1 mapping matrix from big integers: forward = P w and
    # gradient = P^T g, bit for bit on dyadic inputs
    T, B, M = 2, 4, 256
    for seed in range(3):
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed, signed=True)
        A, B0 = bh.params(seed)
        A2, B2 = bh.sign_params(seed)
        L, J = min(Z, d), -(-d // Z)
        R = (M - L) // G + 1
        rows, cols, vals = [], [], []
        for t in range(T):
            for b in range(B):
                s = t * B + b
                for q in range(off[s], off[s + 1]):
                    i = int(idx[q])
                    for k in range(d):
                        j, z = divmod(k, Z)
                        rows.append((b * T + t) * d + k)
                        cols.append(bh.location(A, B0, R, G, T, J, i, t, j) + z)
                        vals.append(bh.sign(A2, B2, T, J, i, t, j))
        P = sp.coo_matrix((vals, (rows, cols)), shape=(B * T * d, M)).tocsr()
        out, bad = o.forward(w, idx, off, B)
        assert bad == -1
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
        np.testing.assert_array_equal(o.grad(idx, off, B, go), P.T @ go.astype(np.float64))


@pytest.mark.parametrize("signed", [False, True])
def test_backward_is_the_adjoint_of_the_forward(signed):
    # <forward(w), g> == <w, grad(g)> for any w, g: the backward of Sec. 2.4 is
    # the transpose of the forward, with or without signs (dyadic: exact)
    cards, idx, off, w, go = _tiny_case(11, T=3, B=8, d=16, M=300, Z=4, G=1, max_bag=5)
    o = OraclePSS(cards, d=16, M=300, Z=4, G=1, seed=5, signed=signed)
    out, _ = o.forward(w, idx, off, 8)
    g = o.grad(idx, off, 8, go)
    lhs = float(np.dot(out.astype(np.float64), go.astype(np.float64)))
    rhs = float(np.dot(w.astype(np.float64), g))
    assert lhs == rhs


def test_signed_grad_at_matches_signed_dense_grad():
    cards, idx, off, w, go = _tiny_case(4, T=2, B=6, d=16, M=512, Z=4, G=2, max_bag=4, dy=False)
    o = OraclePSS(cards, d=16, M=512, Z=4, G=2, seed=8, signed=True)
    g = o.grad(idx, off, 6, go)
    elems = np.flatnonzero(g)
    np.testing.assert_array_equal(o.grad_at(idx, off, 6, go, elems), g[elems])


# --------------------------------------------------------------------------
# circular array (the other reading of the printed range {0..|M_r|}): R = M/G
# starts, and blocks near the end of M wrap to its start
@pytest.mark.parametrize("Z,G,d,signed", [(16, 4, 16, False), (4, 2, 16, False), (32, 4, 16, True),
                                          (3, 1, 10, False)])
def test_circular_forward_and_grad_equal_wrapping_bruteforce_matrix(Z, G, d, signed):
    T, B, M = 2, 4, 64          # small M: many blocks wrap
    wrapped = 0
    for seed in range(4):
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G, max_bag=4)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed, signed=signed, circular=True)
        A, B0 = bh.params(seed)
        A2, B2 = bh.sign_params(seed)
        L, J = min(Z, d), -(-d // Z)
        R = M // G
        assert o.R == R
        rows, cols, vals = [], [], []
        for t in range(T):
            for b in range(B):
                s = t * B + b
                for q in range(off[s], off[s + 1]):
                    i = int(idx[q])
                    for k in range(d):
                        j, z = divmod(k, Z)
                        loc = bh.location(A, B0, R, G, T, J, i, t, j)
                        wrapped += (loc + z) >= M
                        rows.append((b * T + t) * d + k)
                        cols.append((loc + z) % M)
                        vals.append(bh.sign(A2, B2, T, J, i, t, j) if signed else 1)
        P = sp.coo_matrix((vals, (rows, cols)), shape=(B * T * d, M)).tocsr()
        out, bad = o.forward(w, idx, off, B)
        assert bad == -1
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
        np.testing.assert_array_equal(o.grad(idx, off, B, go), P.T @ go.astype(np.float64))
    assert wrapped > 0


def test_circular_with_block_aligned_starts_is_the_plain_mapping():
    # G = L: R = M/L starts either way and no block crosses the end, so the two
    # readings of the range coincide
    cards, idx, off, w, go = _tiny_case(3, T=3, B=8, d=32, M=512, Z=16, G=16, max_bag=5)
    a = OraclePSS(cards, d=32, M=512, Z=16, G=16, seed=2, circular=True)
    b = OraclePSS(cards, d=32, M=512, Z=16, G=16, seed=2)
    assert a.R == b.R
    np.testing.assert_array_equal(a.forward(w, idx, off, 8)[0], b.forward(w, idx, off, 8)[0])
    np.testing.assert_array_equal(a.grad(idx, off, 8, go), b.grad(idx, off, 8, go))


def test_circular_adjoint_sparse_gradient_and_rejection():
    cards, idx, off, w, go = _tiny_case(6, T=3, B=8, d=16, M=96, Z=8, G=4, max_bag=5)
    o = OraclePSS(cards, d=16, M=96, Z=8, G=4, seed=4, circular=True, signed=True)
    out, _ = o.forward(w, idx, off, 8)
    g = o.grad(idx, off, 8, go)
    assert float(np.dot(out.astype(np.float64), go.astype(np.float64))) == float(np.dot(w.astype(np.float64), g))
    elems = np.flatnonzero(g)
    np.testing.assert_array_equal(o.grad_at(idx, off, 8, go, elems), g[elems])
    with pytest.raises(OracleError):
        OraclePSS(cards, d=16, M=98, Z=8, G=4, seed=4, circular=True)


def test_forward_bruteforce_non_dyadic():
    cards, idx, off, w, go = _tiny_case(5, T=3, B=8, d=16, M=300, Z=4, G=1, max_bag=6, dy=False)
    o = OraclePSS(cards, d=16, M=300, Z=4, G=1, seed=9)
    P = _bruteforce_P(cards, idx, off, 8, 16, 300, 4, 1, 9)
    out, _ = o.forward(w, idx, off, 8)
    ref = P @ w.astype(np.float64)
    np.testing.assert_allclose(out, ref, rtol=1e-7, atol=1e-7)
    np.testing.assert_allclose(o.grad(idx, off, 8, go), P.T @ go.astype(np.float64),
                               rtol=1e-12, atol=1e-12)


def test_all_ones_gradient_counts_contributions():
    # The paper's micro-benchmark loss is the sum of all outputs, so the upstream
    # gradient is all ones and g[e] counts how often element e was read.
    cards, idx, off, w, _ = _tiny_case(11, T=3, B=6, d=12, M=200, Z=8, G=2, max_bag=4)
    B, d, M, Z, G, T = 6, 12, 200, 8, 2, 3
    o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=4)
    A, B0 = bh.params(4)
    L, J = min(Z, d), -(-d // Z)
    R = (M - L) // G + 1
    count = np.zeros(M, dtype=np.int64)
    for t in range(T):
        for b in range(B):
            s = t * B + b
            for q in range(off[s], off[s + 1]):
                for j in range(J):
                    loc = bh.location(A, B0, R, G, T, J, int(idx[q]), t, j)
                    for z in range(min(Z, d - j * Z)):
                        count[loc + z] += 1
    g = o.grad(idx, off, B, np.ones(B * T * d, dtype=np.float32))
    np.testing.assert_array_equal(g, count.astype(np.float64))


def test_gradient_mass_invariant():
    w = wl.make_workload("kaggle", B=256)
    o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=0)
    g = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    lengths = np.diff(w.offsets).reshape(w.T, w.B)            # [t][b]
    row_sums = w.grad_out.reshape(w.B, w.T, w.d).astype(np.float64).sum(axis=2)  # [b][t]
    want = float((lengths.T * row_sums).sum())
    assert abs(g.sum() - want) <= 1e-9 * np.abs(w.grad_out).astype(np.float64).sum()


def test_algorithm1_sparse_branch_equals_dense_branch():
    # Algorithm 1: sparse (unique + scatter_add on the unique set) and dense
    # (scatter_add into an M-sized buffer) give the same gradient.
    cards, idx, off, w, go = _tiny_case(21, T=3, B=16, d=16, M=512, Z=4, G=4, max_bag=5,
                                        dy=False)
    B, d, T = 16, 16, 3
    o = OraclePSS(cards, d=d, M=512, Z=4, G=4, seed=2)
    locs, _ = o.locations(idx, off, B)
    # mapping matrix I: element location of every output element read
    I_rows, I_vals = [], []
    for t in range(T):
        for b in range(B):
            s = t * B + b
            for q in range(off[s], off[s + 1]):
                for k in range(d):
                    j, z = divmod(k, 4)
                    I_rows.append(locs[q * o.J + j] + z)
                    I_vals.append(go[(b * T + t) * d + k])
    I_rows = np.asarray(I_rows, dtype=np.int64)
    I_vals = np.asarray(I_vals, dtype=np.float64)
    uniq, inv = np.unique(I_rows, return_inverse=True)
    gs = np.zeros(uniq.shape[0])
    np.add.at(gs, inv, I_vals)
    sparse_dense = np.zeros(512)
    sparse_dense[uniq] = gs
    np.testing.assert_allclose(o.grad(idx, off, B, go), sparse_dense, rtol=1e-12, atol=1e-12)


def test_injective_mapping_is_plain_embedding_bag():
    # Def. 1 with M = E: an injective, row-contiguous mapping makes the pooled
    # gather a plain sum-mode embedding bag.
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    T, B, d, Z = 3, 7, 12, 8
    cards = np.array([5, 9, 4])
    base = np.concatenate([[0], np.cumsum(cards)[:-1]])
    M = int(cards.sum()) * d
    lengths = rng.integers(0, 5, size=T * B)
    off = np.zeros(T * B + 1, dtype=np.int64)
    np.cumsum(lengths, out=off[1:])
    idx = np.concatenate([rng.integers(0, cards[t], size=int(lengths[t * B:(t + 1) * B].sum()))
                          for t in range(T)]).astype(np.int64)
    w = rng.standard_normal(M).astype(np.float32)
    o = OraclePSS(cards, d=d, M=M, Z=Z, G=1, seed=0)
    J = o.J
    locs = np.zeros(idx.shape[0] * J, dtype=np.int64)
    for t in range(T):
        for q in range(off[t * B], off[(t + 1) * B]):
            for j in range(J):
                locs[q * J + j] = (base[t] + idx[q]) * d + j * Z
    out = o.pool(w, locs, off, B, idx.shape[0]).reshape(B, T, d)
    table = torch.from_numpy(w.reshape(-1, d))
    for t in range(T):
        seg = slice(off[t * B], off[(t + 1) * B])
        gid = torch.from_numpy(idx[seg] + base[t])
        offs = torch.from_numpy(off[t * B:(t + 1) * B] - off[t * B])
        ref = torch.nn.functional.embedding_bag(gid, table, offs, mode="sum").numpy()
        np.testing.assert_allclose(out[:, t, :], ref, rtol=1e-6, atol=1e-6)


def test_hashing_trick_special_case():
    # Hashing trick (Sec. 2.5): whole embedding = row h(i) of a 2-D table; this
    # is the mapping with one chunk (Z >= d) and block starts aligned to d.
    rng = np.random.default_rng(8)
    T, B, d = 2, 10, 8
    cards = np.array([100, 37])
    M = 64 * d
    w = rng.standard_normal(M).astype(np.float32)
    lengths = rng.integers(0, 4, size=T * B)
    off = np.zeros(T * B + 1, dtype=np.int64)
    np.cumsum(lengths, out=off[1:])
    idx = np.concatenate([rng.integers(0, cards[t], size=int(lengths[t * B:(t + 1) * B].sum()))
                          for t in range(T)]).astype(np.int64)
    o = OraclePSS(cards, d=d, M=M, Z=d, G=d, seed=5)
    A, B0 = bh.params(5)
    assert o.R == 64
    Mh = w.reshape(64, d).astype(np.float64)
    out, _ = o.forward(w, idx, off, B)
    out = out.reshape(B, T, d)
    for t in range(T):
        for b in range(B):
            s = t * B + b
            ref = np.zeros(d)
            for q in range(off[s], off[s + 1]):
                ref += Mh[bh.bucket(A, B0, 64, int(idx[q]) * T + t)]
            np.testing.assert_allclose(out[b, t], ref.astype(np.float32), rtol=1e-7, atol=1e-7)


def test_edge_cases_empty_partial_chunk_and_single_start():
    # empty bags give zeros; Z not dividing d gives a short last chunk; M = L
    # leaves exactly one possible block start (R = 1).
    cards = np.array([10])
    o = OraclePSS(cards, d=10, M=4, Z=4, G=4, seed=1)
    assert (o.J, o.L, o.R) == (3, 4, 1)
    w = np.arange(4, dtype=np.float32) + 1
    idx = np.array([3, 3, 7], dtype=np.int64)
    off = np.array([0, 0, 3, 3], dtype=np.int64)          # bags: empty, 3 ids, empty
    out, bad = o.forward(w, idx, off, 3)
    assert bad == -1
    out = out.reshape(3, 1, 10)
    np.testing.assert_array_equal(out[0], 0)
    np.testing.assert_array_equal(out[2], 0)
    np.testing.assert_array_equal(out[1, 0], 3 * np.array([1, 2, 3, 4, 1, 2, 3, 4, 1, 2]))


def test_out_of_range_ids_are_skipped_and_reported():
    cards = np.array([5, 5])
    o = OraclePSS(cards, d=4, M=64, Z=4, G=4, seed=1)
    w = np.ones(64, dtype=np.float32)
    idx = np.array([1, 5, -1, 2], dtype=np.int64)
    off = np.array([0, 2, 4], dtype=np.int64)               # B = 1
    out, bad = o.forward(w, idx, off, 1)
    assert bad == 1
    np.testing.assert_array_equal(out.reshape(1, 2, 4)[0, 0], 1.0)
    np.testing.assert_array_equal(out.reshape(1, 2, 4)[0, 1], 1.0)


def test_malformed_offsets_rejected():
    o = OraclePSS(np.array([5]), d=4, M=64, Z=4, G=4, seed=1)
    with pytest.raises(OracleError):
        o.forward(np.ones(64, np.float32), np.array([0, 1], np.int64), np.array([0, 2, 1]), 2)
    with pytest.raises(OracleError):
        o.forward(np.ones(64, np.float32), np.array([0, 1], np.int64), np.array([0, 1, 3]), 2)


def test_init_rejects_bad_sizes():
    with pytest.raises(OracleError):
        OraclePSS(np.array([5]), d=16, M=8, Z=16, G=4)     # no block fits
    with pytest.raises(OracleError):
        OraclePSS(np.array([1 << 60]), d=128, M=1 << 20, Z=32, G=4)  # key beyond P


def test_sgd_matches_torch_sgd():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    w = rng.standard_normal(5000).astype(np.float32)
    g = rng.standard_normal(5000).astype(np.float32)
    g[::7] = 0
    lr = 0.1
    mine = OraclePSS.sgd(w.copy(), g, lr)
    p = torch.nn.Parameter(torch.from_numpy(w.copy()))
    opt = torch.optim.SGD([p], lr=lr)
    p.grad = torch.from_numpy(g.copy())
    opt.step()
    ref = p.detach().numpy()
    # torch may fuse the multiply-add: allow one rounding of the operands
    scale = np.abs(w).astype(np.float64) + lr * np.abs(g).astype(np.float64)
    assert np.all(np.abs(mine.astype(np.float64) - ref) <= 1.2e-7 * scale)
    np.testing.assert_array_equal(mine[::7], w[::7])


def test_sgd_dyadic_exact():
    rng = np.random.default_rng(2)
    w = wl.dyadic(rng, 1000)
    g = wl.dyadic(rng, 1000)
    lr = 0.125
    got = OraclePSS.sgd(w.copy(), g, lr)
    want = (w.astype(np.float64) - lr * g.astype(np.float64))
    np.testing.assert_array_equal(got, want.astype(np.float32))
    assert np.all(got.astype(np.float64) == want)


def test_adagrad_matches_torch_adagrad_three_steps():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    n, lr, eps = 4000, 0.01, 1e-10
    w = rng.standard_normal(n).astype(np.float32) * 0.01
    G = np.zeros(n, dtype=np.float32)
    p = torch.nn.Parameter(torch.from_numpy(w.copy()))
    opt = torch.optim.Adagrad([p], lr=lr, eps=eps, initial_accumulator_value=0.0)
    mine_w = w.copy()
    for _ in range(3):
        g = rng.standard_normal(n).astype(np.float32)
        g[rng.random(n) < 0.2] = 0
        OraclePSS.adagrad(mine_w, G, g, lr, eps)
        p.grad = torch.from_numpy(g.copy())
        opt.step()
    ref_w = p.detach().numpy()
    ref_G = opt.state[p]["sum"].numpy()
    np.testing.assert_allclose(mine_w, ref_w, rtol=1e-6, atol=1e-9)
    np.testing.assert_allclose(G, ref_G, rtol=1e-6, atol=0)


def test_adagrad_first_step_closed_form():
    # From G = 0: w' = w - lr * g / (|g| + eps); for |g| >> eps the quotient
    # rounds to sign(g), so w' = fl(w - lr*sign(g)) exactly.
    rng = np.random.default_rng(4)
    n, lr = 2000, 0.01
    w = rng.standard_normal(n).astype(np.float32) * 0.01
    g = rng.uniform(0.01, 5, n).astype(np.float32) * rng.choice([-1, 1], n).astype(np.float32)
    g[:10] = 0
    G = np.zeros(n, dtype=np.float32)
    w2 = OraclePSS.adagrad(w.copy(), G, g, lr, 1e-10)[0]
    want = (w - np.float32(lr) * np.sign(g)).astype(np.float32)
    np.testing.assert_array_equal(w2[10:], want[10:])
    np.testing.assert_array_equal(w2[:10], w[:10])
    np.testing.assert_array_equal(G[10:], (g[10:] * g[10:]).astype(np.float32))


def test_grad_at_matches_dense_grad():
    w = wl.make_workload("multihot", B=64, M=100_000)
    o = OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=0)
    g = o.grad(w.indices, w.offsets, w.B, w.grad_out)
    rng = np.random.default_rng(0)
    elems = np.unique(np.concatenate([rng.integers(0, w.M, 500), np.flatnonzero(g)[:2000]]))
    ga = o.grad_at(w.indices, w.offsets, w.B, w.grad_out, elems)
    np.testing.assert_allclose(ga, g[elems], rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------
# property-based sweep of the brute-force pin: random tiny shapes, including
# Z > d, Z not dividing d, G > 1 with ragged ranges, empty bags and tables of
# three ids (hypothesis is optional: the GPU hosts do not ship it)
def test_forward_and_grad_equal_bruteforce_matrix_random_shapes():
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=60, deadline=None, derandomize=True)
    @hyp.given(T=st.integers(1, 3), B=st.integers(1, 5), d=st.integers(1, 40),
               Z=st.integers(1, 48), G=st.integers(1, 8), extra=st.integers(0, 300),
               max_bag=st.integers(0, 4), seed=st.integers(0, 2**32 - 1))
    def check(T, B, d, Z, G, extra, max_bag, seed):
        L = min(Z, d)
        M = L + extra
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G, max_bag=max_bag)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed)
        P = _bruteforce_P(cards, idx, off, B, d, M, Z, G, seed)
        out, bad = o.forward(w, idx, off, B)
        assert bad == -1
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
        g = o.grad(idx, off, B, go)
        np.testing.assert_array_equal(g, P.T @ go.astype(np.float64))

    check()


def _bruteforce_P_variant(cards, idx, offsets, B, d, M, Z, G, seed, signed, circular):
    """The +-1 (signed) and wrapping (circular) mapping matrices, from big integers."""
    T = len(cards)
    A, B0 = bh.params(seed)
    A2, B2 = bh.sign_params(seed)
    L, J = min(Z, d), -(-d // Z)
    R = M // G if circular else (M - L) // G + 1
    rows, cols, vals = [], [], []
    for t in range(T):
        for b in range(B):
            s = t * B + b
            for q in range(offsets[s], offsets[s + 1]):
                i = int(idx[q])
                for k in range(d):
                    j, z = divmod(k, Z)
                    loc = bh.location(A, B0, R, G, T, J, i, t, j)
                    rows.append((b * T + t) * d + k)
                    cols.append((loc + z) % M if circular else loc + z)
                    vals.append(bh.sign(A2, B2, T, J, i, t, j) if signed else 1)
    return sp.coo_matrix((vals, (rows, cols)), shape=(B * T * d, M)).tocsr()


def test_signed_and_circular_variants_equal_bruteforce_random_shapes():
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=60, deadline=None, derandomize=True)
    @hyp.given(T=st.integers(1, 3), B=st.integers(1, 5), d=st.integers(1, 40),
               Z=st.integers(1, 48), G=st.integers(1, 8), blocks=st.integers(0, 40),
               max_bag=st.integers(0, 4), seed=st.integers(0, 2**32 - 1),
               signed=st.booleans(), circular=st.booleans())
    def check(T, B, d, Z, G, blocks, max_bag, seed, signed, circular):
        L = min(Z, d)
        # circular: G divides M; both readings: M >= L
        M = G * (-(-L // G) + blocks) if circular else L + blocks * G
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G, max_bag=max_bag)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed, signed=signed, circular=circular)
        P = _bruteforce_P_variant(cards, idx, off, B, d, M, Z, G, seed, signed, circular)
        out, bad = o.forward(w, idx, off, B)
        assert bad == -1
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
        np.testing.assert_array_equal(o.grad(idx, off, B, go), P.T @ go.astype(np.float64))

    check()


@pytest.mark.parametrize("signed", [False, True])
def test_scatter_and_signs_entry_points_equal_bruteforce(signed):
    # the lower-level entry points: signs() per (id, chunk) from big integers,
    # scatter() of explicit locations (and signs) equal to P^T g, and pool()
    # of the same equal to P w
    T, B, d, M, Z, G = 3, 5, 20, 400, 8, 2
    for seed in range(3):
        cards, idx, off, w, go = _tiny_case(seed, T=T, B=B, d=d, M=M, Z=Z, G=G, max_bag=4)
        o = OraclePSS(cards, d=d, M=M, Z=Z, G=G, seed=seed, signed=signed)
        A, B0 = bh.params(seed)
        A2, B2 = bh.sign_params(seed)
        J, L = -(-d // Z), min(Z, d)
        R = (M - L) // G + 1
        locs = np.zeros(idx.shape[0] * J, dtype=np.int64)
        sg = np.zeros(idx.shape[0] * J, dtype=np.int64)
        for t in range(T):
            for q in range(off[t * B], off[(t + 1) * B]):
                for j in range(J):
                    locs[q * J + j] = bh.location(A, B0, R, G, T, J, int(idx[q]), t, j)
                    sg[q * J + j] = bh.sign(A2, B2, T, J, int(idx[q]), t, j)
        if signed:
            np.testing.assert_array_equal(o.signs(idx, off, B).astype(np.int64), sg)
        P = _bruteforce_P_variant(cards, idx, off, B, d, M, Z, G, seed, signed, False)
        s8 = sg.astype(np.int8) if signed else None
        g = o.scatter(locs, off, B, idx.shape[0], go, signs=s8)
        np.testing.assert_array_equal(g, P.T @ go.astype(np.float64))
        out = o.pool(w, locs, off, B, idx.shape[0], signs=s8)
        np.testing.assert_array_equal(out, (P @ w.astype(np.float64)).astype(np.float32))
