// CUDA kernels of libpss (sm_103a): location hash, fused hash + gather +
// sum-pool forward, hash + vector-atomic backward scatter, and the optimizer
// passes over the shared array.
//
// Work decomposition shared by the forward and backward kernels: one GROUP of
// gs lanes per bag (gs = 32 for d >= 128 in float4 columns, 16 for d = 64, 4
// for d = 16), so a warp always moves whole 16-byte columns and a bag row is
// written with one coalesced store per lane.  Groups walk bag slots in
// table-major order with a grid-stride loop, so neighbouring groups read
// neighbouring offsets/indices.
#include <climits>
#include <type_traits>

#include "pss_device.cuh"
#include "pss_internal.h"

namespace pss {

namespace {

// ---------------------------------------------------------------------------
// Location hash only: locs[q*J + j] (the mapping matrix of Algorithm 1).
__global__ void __launch_bounds__(kThreads)
k_locations(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
            const int64_t* __restrict__ off, int64_t B, uint64_t Binv, int64_t* __restrict__ locs,
            DevError* err) {
    pdl_prologue();
    const int64_t nbags = (int64_t)p.T * B;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s < nbags; s += stride) {
        int t;
        int64_t b, q0, q1;
        split_slot(s, B, Binv, t, b);
        if (!bag_range(off, s, nnz, q0, q1)) record_bad_offsets(err);
        const uint64_t card = (uint64_t)__ldg(p.cards + t);
        for (int64_t q = q0; q < q1; ++q) {
            const int64_t id = __ldg(idx + q);
            if ((uint64_t)id >= card) {
                record_bad_id(err, q);
                for (int j = 0; j < p.J; ++j) locs[q * p.J + j] = -1;
                continue;
            }
            const uint64_t kb = hash_key(p, (uint64_t)id, t, 0);
            for (int j = 0; j < p.J; ++j)
                locs[q * p.J + j] = (int64_t)((uint64_t)p.G * hash_bucket(p, kb + j));
        }
    }
}

// ---------------------------------------------------------------------------
// Optimizer arithmetic, one IEEE operation at a time (no contraction):
//   SGD:     w <- w - lr*g
//   Adagrad: G <- G + g*g;  w <- w - lr * (g / (sqrt(G) + eps))
__device__ __forceinline__ void sgd_elem(float& w, float g, float lr) {
    w = __fsub_rn(w, __fmul_rn(lr, g));
}
__device__ __forceinline__ void adagrad_elem(float& w, float& Ga, float g, float lr, float eps) {
    const float Gn = __fadd_rn(Ga, __fmul_rn(g, g));
    const float den = __fadd_rn(__fsqrt_rn(Gn), eps);
    const float q = __fdiv_rn(g, den);
    w = __fsub_rn(w, __fmul_rn(lr, q));
    Ga = Gn;
}

template <typename GT>
__device__ __forceinline__ bool load4_nonzero(GT* g, int64_t i, float (&gv)[4]);
template <>
__device__ __forceinline__ bool load4_nonzero<float>(float* g, int64_t i, float (&gv)[4]) {
    const float4 v = reinterpret_cast<const float4*>(g)[i];
    gv[0] = v.x; gv[1] = v.y; gv[2] = v.z; gv[3] = v.w;
    return v.x != 0.f || v.y != 0.f || v.z != 0.f || v.w != 0.f;
}
template <>
__device__ __forceinline__ bool load4_nonzero<double>(double* g, int64_t i, float (&gv)[4]) {
    const double2 a = reinterpret_cast<const double2*>(g)[2 * i];
    const double2 b = reinterpret_cast<const double2*>(g)[2 * i + 1];
    gv[0] = to_f32(a.x); gv[1] = to_f32(a.y); gv[2] = to_f32(b.x); gv[3] = to_f32(b.y);
    return nonzero(a.x) || nonzero(a.y) || nonzero(b.x) || nonzero(b.y);
}
__device__ __forceinline__ void zero4(float* g, int64_t i) {
    reinterpret_cast<float4*>(g)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
}
__device__ __forceinline__ void zero4(double* g, int64_t i) {
    reinterpret_cast<double2*>(g)[2 * i] = make_double2(0.0, 0.0);
    reinterpret_cast<double2*>(g)[2 * i + 1] = make_double2(0.0, 0.0);
}

// Dense pass over M: apply the step where the (rounded) gradient is non-zero
// and return the accumulator to zero.
template <bool ADA, typename GT>
__global__ void __launch_bounds__(kThreads)
k_update_dense(float* __restrict__ w, float* __restrict__ Ga, GT* __restrict__ g, int64_t M,
               float lr, float eps) {
    pdl_prologue();
    const int64_t n4 = M >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    float4* w4 = reinterpret_cast<float4*>(w);
    float4* G4 = reinterpret_cast<float4*>(Ga);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float gv[4];
        if (!load4_nonzero(g, i, gv)) continue;
        float4 wv = w4[i];
        float* wp = reinterpret_cast<float*>(&wv);
        if (ADA) {
            float4 Gv = G4[i];
            float* Gp = reinterpret_cast<float*>(&Gv);
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (gv[c] != 0.f) adagrad_elem(wp[c], Gp[c], gv[c], lr, eps);
            G4[i] = Gv;
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (gv[c] != 0.f) sgd_elem(wp[c], gv[c], lr);
        }
        w4[i] = wv;
        zero4(g, i);
    }
    for (int64_t e = n4 * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < M; e += stride) {
        if (!nonzero(g[e])) continue;
        const float gv = to_f32(g[e]);
        if (gv != 0.f) {
            if (ADA) adagrad_elem(w[e], Ga[e], gv, lr, eps);
            else sgd_elem(w[e], gv, lr);
        }
        g[e] = (GT)0;
    }
}

// Circular array: the gradient accumulator has L elements past M that stand
// for M[0 .. L) (blocks near the end wrap there); fold them into the head and
// clear them.
template <typename GT>
__global__ void __launch_bounds__(kThreads) k_fold_tail(GT* __restrict__ g, int64_t M, int L) {
    pdl_prologue();
    for (int z = blockIdx.x * blockDim.x + threadIdx.x; z < L; z += gridDim.x * blockDim.x) {
        const GT v = g[M + z];
        if (nonzero(v)) {
            g[z] += v;
            g[M + z] = (GT)0;
        }
    }
}

// Conversion check: the integer fp32 <-> fp64 conversions of the accumulation
// path applied to n values.
__global__ void __launch_bounds__(kThreads)
k_convert(int direction, const void* __restrict__ in, void* __restrict__ out, int64_t n) {
    pdl_prologue();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        if (direction == 0)
            static_cast<double*>(out)[i] = widen(static_cast<const float*>(in)[i]);
        else
            static_cast<float*>(out)[i] = narrow(static_cast<const double*>(in)[i]);
    }
}

// Gradient export: out[e] = fp32(g[e]) and g[e] = 0, over all of M.
__global__ void __launch_bounds__(kThreads)
k_grad_export(double* __restrict__ g, float* __restrict__ out, int64_t M) {
    pdl_prologue();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < M; e += stride) {
        const double v = g[e];
        out[e] = to_f32(v);
        if (nonzero(v)) g[e] = 0.0;
    }
}

// Touched-block pass: one warp per kTU distinct block starts x at a time
// (from the list), their loads in flight together.  Element e = x*G + z
// belongs to the LAST marked start at or below it (no marked bucket in
// (x, x + z/G]), so every element is updated exactly once and without atomics
// even though blocks overlap when G < L.
constexpr int kTU = 4;

__device__ __forceinline__ bool owns(const uint32_t* __restrict__ bitmap, uint64_t x, int nb) {
    for (int m0 = 1; m0 <= nb; m0 += 32) {
        const uint64_t y = x + (uint64_t)m0;
        const uint64_t w0 = bitmap[y >> 5];
        const uint64_t w1 = bitmap[(y >> 5) + 1];
        const uint64_t win = ((w1 << 32) | w0) >> (y & 31);
        const int cnt = (nb - m0 + 1) < 32 ? (nb - m0 + 1) : 32;
        const uint64_t mask = (cnt >= 32) ? 0xffffffffull : ((1ull << cnt) - 1);
        if (win & mask) return false;
    }
    return true;
}

template <bool ADA, typename GT>
__global__ void __launch_bounds__(kThreads)
k_update_touched(float* __restrict__ w, float* __restrict__ Ga, GT* __restrict__ g,
                 Touched tc, int64_t G, int L, float lr, float eps) {
    pdl_prologue();
    const int lane = threadIdx.x & 31;
    unsigned long long n = *tc.count;
    if ((int64_t)n > tc.cap) n = (unsigned long long)tc.cap;
    const int64_t stride = (int64_t)gridDim.x * kWarps * kTU;
    for (int64_t it = ((int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5)) * kTU; it < (int64_t)n;
         it += stride) {
        uint64_t x[kTU];
        bool valid[kTU];
#pragma unroll
        for (int u = 0; u < kTU; ++u) {
            valid[u] = it + u < (int64_t)n;
            x[u] = valid[u] ? (uint64_t)tc.list[it + u] : 0ull;
        }
        for (int z = lane; z < L; z += 32) {
            const int nb = (int)(z / G);   // following starts that could also cover e
            bool own[kTU];
            GT raw[kTU];
#pragma unroll
            for (int u = 0; u < kTU; ++u) own[u] = valid[u] && owns(tc.bitmap, x[u], nb);
#pragma unroll
            for (int u = 0; u < kTU; ++u) raw[u] = own[u] ? g[(int64_t)x[u] * G + z] : (GT)0;
            float wv[kTU], gav[kTU];
#pragma unroll
            for (int u = 0; u < kTU; ++u) {
                wv[u] = gav[u] = 0.f;
                if (nonzero(raw[u])) {
                    const int64_t e = (int64_t)x[u] * G + z;
                    wv[u] = w[e];
                    if (ADA) gav[u] = Ga[e];
                }
            }
#pragma unroll
            for (int u = 0; u < kTU; ++u) {
                if (!nonzero(raw[u])) continue;
                const int64_t e = (int64_t)x[u] * G + z;
                const float gv = to_f32(raw[u]);
                if (gv != 0.f) {
                    if (ADA) {
                        adagrad_elem(wv[u], gav[u], gv, lr, eps);
                        Ga[e] = gav[u];
                    } else {
                        sgd_elem(wv[u], gv, lr);
                    }
                    w[e] = wv[u];
                }
                g[e] = (GT)0;
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads) k_touched_clear(Touched tc) {
    pdl_prologue();
    unsigned long long n = *tc.count;
    if ((int64_t)n > tc.cap) n = (unsigned long long)tc.cap;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < (int64_t)n; i += stride)
        tc.bitmap[(uint64_t)tc.list[i] >> 5] = 0u;
}

template <bool ADA, typename GT>
cudaError_t update_dense_inst(float* w, float* Ga, GT* g, int64_t M, float lr, float eps,
                              int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_update_dense<ADA, GT>, sm_count, ((M >> 2) + kThreads) / kThreads);
    return launch_k(k_update_dense<ADA, GT>, dim3(grid), dim3(kThreads), 0, st, w, Ga, g, M, lr,
                    eps);
}

template <bool ADA, typename GT>
cudaError_t update_touched_inst(float* w, float* Ga, GT* g, const Touched& tc, int64_t G,
                                int32_t L, float lr, float eps, int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_update_touched<ADA, GT>, sm_count,
                              (tc.cap + kWarps * kTU - 1) / (kWarps * kTU));
    return launch_k(k_update_touched<ADA, GT>, dim3(grid), dim3(kThreads), 0, st, w, Ga, g, tc, G,
                    L, lr, eps);
}

}  // namespace

RowLayout choose_layout(int d, int Z, int64_t G) {
    RowLayout r;
    r.vw = (d % 4 == 0 && Z % 4 == 0 && G % 4 == 0) ? 4 : 1;
    const int V = d / r.vw;
    if (V <= 32) {
        r.log2gs = ceil_log2(V);
        r.kc = 1;
    } else {
        r.log2gs = 5;
        r.kc = 1 << ceil_log2((V + 31) / 32);
    }
    return r;
}

cudaError_t launch_locations(const DevParams& p, const int64_t* idx, int64_t nnz,
                             const int64_t* off, int64_t B, int64_t* locs, DevError* err,
                             int sm_count, cudaStream_t st) {
    const int64_t nbags = (int64_t)p.T * B;
    const int grid = grid_for(k_locations, sm_count, (nbags + kThreads - 1) / kThreads);
    return launch_k(k_locations, dim3(grid), dim3(kThreads), 0, st, p, idx, nnz, off, B,
                    UINT64_MAX / (uint64_t)B, locs, err);
}

cudaError_t launch_update_dense(bool adagrad, float* w, float* Ga, float* g, int64_t M, float lr,
                                float eps, int sm_count, cudaStream_t st) {
    return adagrad ? update_dense_inst<true, float>(w, Ga, g, M, lr, eps, sm_count, st)
                   : update_dense_inst<false, float>(w, Ga, g, M, lr, eps, sm_count, st);
}

cudaError_t launch_update_dense64(bool adagrad, float* w, float* Ga, double* g, int64_t M,
                                  float lr, float eps, int sm_count, cudaStream_t st) {
    return adagrad ? update_dense_inst<true, double>(w, Ga, g, M, lr, eps, sm_count, st)
                   : update_dense_inst<false, double>(w, Ga, g, M, lr, eps, sm_count, st);
}

cudaError_t launch_update_touched(bool adagrad, float* w, float* Ga, float* g, const Touched& tc,
                                  int64_t G, int32_t L, float lr, float eps, int sm_count,
                                  cudaStream_t st) {
    return adagrad ? update_touched_inst<true, float>(w, Ga, g, tc, G, L, lr, eps, sm_count, st)
                   : update_touched_inst<false, float>(w, Ga, g, tc, G, L, lr, eps, sm_count, st);
}

cudaError_t launch_update_touched64(bool adagrad, float* w, float* Ga, double* g,
                                    const Touched& tc, int64_t G, int32_t L, float lr, float eps,
                                    int sm_count, cudaStream_t st) {
    return adagrad ? update_touched_inst<true, double>(w, Ga, g, tc, G, L, lr, eps, sm_count, st)
                   : update_touched_inst<false, double>(w, Ga, g, tc, G, L, lr, eps, sm_count, st);
}

cudaError_t launch_grad_export(double* g, float* out, int64_t M, int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_grad_export, sm_count, (M + kThreads - 1) / kThreads);
    return launch_k(k_grad_export, dim3(grid), dim3(kThreads), 0, st, g, out, M);
}

cudaError_t launch_fold_tail(double* g64, float* g32, int64_t M, int L, cudaStream_t st) {
    const int grid = (L + kThreads - 1) / kThreads;
    if (g64) return launch_k(k_fold_tail<double>, dim3(grid), dim3(kThreads), 0, st, g64, M, L);
    return launch_k(k_fold_tail<float>, dim3(grid), dim3(kThreads), 0, st, g32, M, L);
}

cudaError_t launch_convert(int direction, const void* in, void* out, int64_t n, int sm_count,
                           cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int grid = grid_for(k_convert, sm_count, (n + kThreads - 1) / kThreads);
    return launch_k(k_convert, dim3(grid), dim3(kThreads), 0, st, direction, in, out, n);
}

cudaError_t launch_touched_clear(const Touched& tc, int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_touched_clear, sm_count, (tc.cap + kThreads - 1) / kThreads);
    const cudaError_t e = launch_k(k_touched_clear, dim3(grid), dim3(kThreads), 0, st, tc);
    if (e != cudaSuccess) return e;
    return cudaMemsetAsync(tc.count, 0, sizeof(unsigned long long), st);
}

}  // namespace pss
