"""Helpers shared by the GPU parity tests: building handles from workloads and
the condition-aware tolerances.

Tolerances (derived from fp32 summation error; Higham, "Accuracy and Stability
of Numerical Algorithms", Sec. 4.2: a recursive fp32 sum of n terms has error
at most (n-1) u sum|x_i|, u = 2^-24, in ANY order):
  * forward output k of a bag:   |gpu - ref| <= 1e-6 * sum_i |x_i|
    (the kernel uses compensated summation, whose bound is 2u sum|x_i| for any n)
  * gradient element e:          |gpu - ref| <= 1e-5 * A_e,  A_e = sum |contributions to e|
  * SGD:       |w'_gpu - w'_ref| <= 1e-5 * max(|w'_ref|, lr * A_e)
  * Adagrad:   G' = G + g^2 and w' = w - lr g / (sqrt(G') + eps) propagate the
    gradient error dg <= 1e-5 A_e through |dG'| <= 2|g| dg + dg^2 and
    |dw'| <= lr * dg / sqrt(G'), plus a few fp32 roundings of the operands.
"""
import numpy as np

import oracle
from paper_2207_10731_gb300 import binding, workloads as wl

U32 = 2.0 ** -24
FWD_TOL = 1e-6
GRAD_TOL = 1e-5


def torch():
    import torch as _t
    return _t


def cuda(a):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.detach().cpu().numpy()


def make_pair(w: wl.Workload, opt=None, seed=None):
    """(GPU handle with w0 loaded, oracle instance) for a workload."""
    opt = opt or w.opt
    seed = w.seed if seed is None else seed
    h = binding.PSS(w.cards, dim=w.d, M=w.M, Z=w.Z, G=w.G, seed=seed, optimizer=opt, eps=w.eps)
    if w.w0 is not None:
        h.set_weights(cuda(w.w0))
    else:
        t = torch()
        base = cuda(w.w0_base)
        reps = -(-w.M // base.numel())
        full = base.repeat(reps)[: w.M].contiguous()
        h.set_weights(full)
        t.cuda.synchronize()
        del full, base
        t.cuda.empty_cache()
    o = oracle.OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=seed)
    return h, o


def check_forward(out_gpu, out_ref, abs_pool, tol=FWD_TOL, what="forward"):
    err = np.abs(out_gpu.astype(np.float64) - out_ref.astype(np.float64))
    bound = tol * abs_pool.astype(np.float64)
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} elements beyond tolerance; worst "
                           f"err {err[bad].max():.3e} vs bound {bound[bad][np.argmax(err[bad])]:.3e}")


def check_grad(g_gpu, g_ref, A, tol=GRAD_TOL, what="grad"):
    err = np.abs(g_gpu.astype(np.float64) - g_ref)
    bound = tol * A
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} elements beyond tolerance; worst err "
                           f"{err[bad].max():.3e}")


def check_sgd(w_gpu, w_ref, A, lr, tol=GRAD_TOL, what="sgd"):
    err = np.abs(w_gpu.astype(np.float64) - w_ref.astype(np.float64))
    bound = tol * np.maximum(np.abs(w_ref.astype(np.float64)), lr * A) + 2 * U32 * np.abs(w_ref)
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} elements beyond tolerance; worst err "
                           f"{err[bad].max():.3e}")


def check_adagrad(w_gpu, G_gpu, w_ref, G_ref, g_ref, A, lr, tol=GRAD_TOL, what="adagrad"):
    dg = tol * A
    g64 = np.abs(g_ref.astype(np.float64))
    Gr = G_ref.astype(np.float64)
    errG = np.abs(G_gpu.astype(np.float64) - Gr)
    boundG = 2 * g64 * dg + dg * dg + 4 * U32 * Gr
    badG = errG > boundG
    assert not badG.any(), f"{what}: accumulator off at {int(badG.sum())} elements"
    with np.errstate(divide="ignore", invalid="ignore"):
        dw = np.where(Gr > 0, lr * dg / np.sqrt(Gr), np.inf)
    dw = np.where(dg == 0, 0.0, dw)
    errw = np.abs(w_gpu.astype(np.float64) - w_ref.astype(np.float64))
    boundw = dw + 8 * U32 * (np.abs(w_ref.astype(np.float64)) + lr)
    badw = errw > boundw
    assert not badw.any(), (f"{what}: weights off at {int(badw.sum())} elements; worst err "
                            f"{errw[badw].max():.3e}")


def ctypes_ptr(t):
    import ctypes
    return ctypes.c_void_p(int(t.data_ptr()))
