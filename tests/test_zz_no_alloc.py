"""pss_grad_noalloc: the allocation-free gradient entry point.

It exists for callers that cannot call cudaMalloc -- code embedded in a host
framework that owns the whole device-memory budget, or latency-critical code
that cannot accept an allocation's implicit synchronisation.  Its scratch is a
fixed-size device array inside the library.  These tests call it through the C
ABI and compare it with the CPU oracle's gradient on two calls in a row (the
second call must not see the first call's leftovers), within the gradient
tolerance the other parity tests use, and with the handle-based
pss_backward_grad on the same inputs.
"""
import ctypes

import numpy as np
import pytest

from paper_2207_10731_gb300 import binding, workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

MAX_M = 1 << 22


def _call(lib, w, indices, offsets, grad_out, grad, first_bad, stream):
    cards = np.ascontiguousarray(w.cards, dtype=np.int64)
    return lib.pss_grad_noalloc(ctypes.c_void_p(cards.ctypes.data), w.T, w.d, w.M, w.Z, w.G,
                                ctypes.c_uint64(w.seed), gu.ctypes_ptr(indices), indices.numel(),
                                gu.ctypes_ptr(offsets), w.B, gu.ctypes_ptr(grad_out),
                                gu.ctypes_ptr(grad), gu.ctypes_ptr(first_bad),
                                ctypes.c_void_p(int(stream.cuda_stream)))


# 300 tables: the table sizes reach the device in two launches of 256
@pytest.mark.parametrize("name,B,over", [("kaggle", 2048, {}), ("tb", 4096, {}),
                                         ("multihot", 1024, {}), ("tiny", 64, {"T": 300})],
                         ids=["kaggle", "tb", "multihot", "tiny-300-tables"])
def test_noalloc_gradient_matches_oracle_two_calls(name, B, over):
    t = gu.torch()
    lib = binding.load_library()
    stream = t.cuda.current_stream()
    for batch in (0, 1):
        w = wl.make_workload(name, B=B, batch=batch, **over)
        assert w.M <= MAX_M
        h, o = gu.make_pair(w)
        idx, off, go = gu.cuda(w.indices), gu.cuda(w.offsets), gu.cuda(w.grad_out)
        h.forward(idx, off, w.B)
        g_handle = gu.host(h.backward_grad(go)).astype(np.float64)
        h.close()
        grad = t.full((w.M,), float("nan"), dtype=t.float32, device="cuda")
        first_bad = t.zeros(1, dtype=t.int64, device="cuda")
        assert _call(lib, w, idx, off, go, grad, first_bad, stream) == binding.PSS_OK
        t.cuda.synchronize()
        g_ref = o.grad(w.indices, w.offsets, w.B, w.grad_out)
        A = o.grad(w.indices, w.offsets, w.B, np.abs(w.grad_out))
        g = gu.host(grad)
        gu.check_grad(g, g_ref, A, what=f"noalloc {name} batch {batch} vs oracle")
        gu.check_grad(g, g_handle, 2 * A, what=f"noalloc {name} batch {batch} vs handle")
        assert int(first_bad.item()) == -1


def test_noalloc_reports_bad_ids_and_rejects_what_it_cannot_serve():
    t = gu.torch()
    lib = binding.load_library()
    stream = t.cuda.current_stream()
    w = wl.make_workload("tiny")
    idx = w.indices.copy()
    idx[50] = 10_000
    grad = t.empty(w.M, dtype=t.float32, device="cuda")
    first_bad = t.zeros(1, dtype=t.int64, device="cuda")
    d_idx, d_off, d_go = gu.cuda(idx), gu.cuda(w.offsets), gu.cuda(w.grad_out)
    assert _call(lib, w, d_idx, d_off, d_go, grad, first_bad, stream) == binding.PSS_OK
    t.cuda.synchronize()
    assert int(first_bad.item()) == 50
    # host batch buffers are not staged (that would allocate): rejected
    rc = _call(lib, w, t.from_numpy(idx), d_off, d_go, grad, first_bad, stream)
    assert rc == binding.PSS_ERR_INVALID_ARG
    # beyond the fixed scratch: a clear capacity error, nothing queued
    big = wl.make_workload("tiny")
    big.M = MAX_M + 1
    rc = _call(lib, big, d_idx, d_off, d_go, grad, first_bad, stream)
    assert rc == binding.PSS_ERR_CAPACITY
    assert "capacity" in binding.status_string(rc)
