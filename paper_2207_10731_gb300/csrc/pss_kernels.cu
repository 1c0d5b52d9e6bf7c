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

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

int ceil_log2(int v) {
    int l = 0;
    while ((1 << l) < v) ++l;
    return l;
}

template <typename K>
int grid_for(K kernel, int sm_count, int64_t work_blocks) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, 0) != cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    int64_t g = (int64_t)sm_count * per_sm;
    if (work_blocks < g) g = work_blocks;
    if (g < 1) g = 1;
    return (int)g;
}

// Per-lane column description inside one bag row.
template <int VW, int KC>
struct Cols {
    int j[KC];     // chunk of the column
    int z[KC];     // offset of the column inside its chunk
    bool v[KC];    // column exists (d not a multiple of the group width)
    int e[KC];     // element offset of the column in the row
    __device__ __forceinline__ Cols(const DevParams& p, int lg, int gs) {
        const int V = p.d / VW;
#pragma unroll
        for (int k = 0; k < KC; ++k) {
            const int c = lg + k * gs;
            v[k] = c < V;
            e[k] = c * VW;
            j[k] = e[k] / p.Z;
            z[k] = e[k] - j[k] * p.Z;
        }
    }
};

template <int VW>
struct Vec;
template <>
struct Vec<4> {
    using T = float4;
    static __device__ __forceinline__ float4 ldg(const float* p) {
        return __ldg(reinterpret_cast<const float4*>(p));
    }
    static __device__ __forceinline__ float4 ldcs(const float* p) {
        return __ldcs(reinterpret_cast<const float4*>(p));
    }
    static __device__ __forceinline__ void stcs(float* p, float4 v) {
        __stcs(reinterpret_cast<float4*>(p), v);
    }
    static __device__ __forceinline__ void red(float* p, float4 v) { red_add_v4(p, v); }
    static __device__ __forceinline__ float get(const float4& v, int i) {
        return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
    }
    static __device__ __forceinline__ void set(float4& v, int i, float x) {
        if (i == 0) v.x = x; else if (i == 1) v.y = x; else if (i == 2) v.z = x; else v.w = x;
    }
    static __device__ __forceinline__ float4 scale(float4 v, float s) {
        return make_float4(__fmul_rn(v.x, s), __fmul_rn(v.y, s), __fmul_rn(v.z, s),
                           __fmul_rn(v.w, s));
    }
};
template <>
struct Vec<1> {
    using T = float;
    static __device__ __forceinline__ float ldg(const float* p) { return __ldg(p); }
    static __device__ __forceinline__ float ldcs(const float* p) { return __ldcs(p); }
    static __device__ __forceinline__ void stcs(float* p, float v) { __stcs(p, v); }
    static __device__ __forceinline__ void red(float* p, float v) { red_add_f32(p, v); }
    static __device__ __forceinline__ float get(const float& v, int) { return v; }
    static __device__ __forceinline__ void set(float& v, int, float x) { v = x; }
    static __device__ __forceinline__ float scale(float v, float s) { return __fmul_rn(v, s); }
};

// Bag slot s -> (table t, row b) for s = t*B + b, with Binv = floor((2^64-1)/B):
// umulhi(s, Binv) is t or t-1 (same argument as the hash's "mod R").
__device__ __forceinline__ void split_slot(int64_t s, int64_t B, uint64_t Binv, int& t, int64_t& b) {
    uint64_t q = __umul64hi((uint64_t)s, Binv);
    uint64_t r = (uint64_t)s - q * (uint64_t)B;
    if (r >= (uint64_t)B) {
        ++q;
        r -= (uint64_t)B;
    }
    t = (int)q;
    b = (int64_t)r;
}

// Reduction of one VW-wide column into an fp32 or fp64 accumulator.
template <int VW, typename AT>
struct Acc;
template <int VW>
struct Acc<VW, float> {
    static __device__ __forceinline__ void red(float* p, typename Vec<VW>::T v) { Vec<VW>::red(p, v); }
};
template <>
struct Acc<4, double> {
    static __device__ __forceinline__ void red(double* p, float4 v) {
        red_add_f64(p + 0, (double)v.x);
        red_add_f64(p + 1, (double)v.y);
        red_add_f64(p + 2, (double)v.z);
        red_add_f64(p + 3, (double)v.w);
    }
};
template <>
struct Acc<1, double> {
    static __device__ __forceinline__ void red(double* p, float v) { red_add_f64(p, (double)v); }
};

// Accumulator element -> fp32 gradient (rounded once, to nearest).
__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(double v) { return __double2float_rn(v); }

__device__ __forceinline__ bool bag_range(const int64_t* __restrict__ off, int64_t s, int64_t nnz,
                                          int64_t& q0, int64_t& q1) {
    q0 = __ldg(off + s);
    q1 = __ldg(off + s + 1);
    if (q0 < 0 || q1 < q0 || q1 > nnz) {
        q0 = q1 = 0;
        return false;
    }
    return true;
}

// ---------------------------------------------------------------------------
// Location hash only: locs[q*J + j] (the mapping matrix of Algorithm 1).
__global__ void __launch_bounds__(kThreads)
k_locations(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
            const int64_t* __restrict__ off, int64_t B, uint64_t Binv, int64_t* __restrict__ locs,
            DevError* err) {
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
// Forward: out[b][t][:] = sum over ids of bag (t,b) of the hashed blocks.
template <int VW, int KC>
__global__ void __launch_bounds__(kThreads)
k_forward(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
          const int64_t* __restrict__ off, int64_t B, uint64_t Binv, const float* __restrict__ w,
          float* __restrict__ out, DevError* err, int log2gs) {
    using V = Vec<VW>;
    const int lane = threadIdx.x & 31;
    const int gs = 1 << log2gs;
    const int lg = lane & (gs - 1);
    const int ng = 32 >> log2gs;
    const Cols<VW, KC> col(p, lg, gs);
    const uint64_t G = (uint64_t)p.G;
    const int64_t nbags = (int64_t)p.T * B;
    const int64_t stride = (int64_t)gridDim.x * kWarps * ng;
    int64_t s = ((int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5)) * ng + (lane >> log2gs);
    for (; s < nbags; s += stride) {
        int t;
        int64_t b, q0, q1;
        split_slot(s, B, Binv, t, b);
        if (!bag_range(off, s, nnz, q0, q1) && lg == 0) record_bad_offsets(err);
        const uint64_t card = (uint64_t)__ldg(p.cards + t);
        float acc[KC][VW], cmp[KC][VW];
#pragma unroll
        for (int k = 0; k < KC; ++k)
#pragma unroll
            for (int i = 0; i < VW; ++i) acc[k][i] = cmp[k][i] = 0.f;
        for (int64_t q = q0; q < q1; ++q) {
            const int64_t id = __ldg(idx + q);
            if ((uint64_t)id >= card) {
                if (lg == 0) record_bad_id(err, q);
                continue;
            }
            const uint64_t kb = hash_key(p, (uint64_t)id, t, 0);
#pragma unroll
            for (int k = 0; k < KC; ++k) {
                if (!col.v[k]) continue;
                const uint64_t loc = G * hash_bucket(p, kb + col.j[k]);
                const typename V::T x = V::ldg(w + loc + col.z[k]);
#pragma unroll
                for (int i = 0; i < VW; ++i) kahan_add(acc[k][i], cmp[k][i], V::get(x, i));
            }
        }
        float* orow = out + (b * p.T + t) * (int64_t)p.d;
#pragma unroll
        for (int k = 0; k < KC; ++k) {
            if (!col.v[k]) continue;
            typename V::T o;
#pragma unroll
            for (int i = 0; i < VW; ++i) V::set(o, i, acc[k][i]);
            V::stcs(orow + col.e[k], o);
        }
    }
}

__device__ __forceinline__ void mark_touched(const Touched& tc, uint64_t x) {
    uint32_t* wp = tc.bitmap + (x >> 5);
    const uint32_t bit = 1u << (x & 31);
    if (*reinterpret_cast<volatile uint32_t*>(wp) & bit) return;
    const uint32_t old = atomicOr(wp, bit);
    if (!(old & bit)) {
        const unsigned long long slot = atomicAdd(tc.count, 1ULL);
        if ((int64_t)slot < tc.cap) tc.list[slot] = (int64_t)x;
    }
}

// ---------------------------------------------------------------------------
// Backward scatter (dense branch of Algorithm 1): for every id of every bag,
// add scale * grad_out row chunk j into target[loc(t,i,j) + z].  AT = double
// accumulates in fp64 (one scalar reduction per element: the result is the
// exact sum up to n*2^-53 relative, rounded once later); AT = float uses 16-byte
// fp32 vector reductions (recursive fp32 summation in atomic order).  With an
// fp32 target = M and scale = -lr this is the whole SGD step.  TOUCH also
// records every distinct block start in the touched bitmap/list.
template <int VW, int KC, bool TOUCH, typename AT>
__global__ void __launch_bounds__(kThreads)
k_scatter(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
          const int64_t* __restrict__ off, int64_t B, uint64_t Binv, const float* __restrict__ gout,
          float scale, AT* target, Touched tc, DevError* err, int log2gs) {
    using V = Vec<VW>;
    const int lane = threadIdx.x & 31;
    const int gs = 1 << log2gs;
    const int lg = lane & (gs - 1);
    const int ng = 32 >> log2gs;
    const Cols<VW, KC> col(p, lg, gs);
    const uint64_t G = (uint64_t)p.G;
    const int64_t nbags = (int64_t)p.T * B;
    const int64_t stride = (int64_t)gridDim.x * kWarps * ng;
    int64_t s = ((int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5)) * ng + (lane >> log2gs);
    for (; s < nbags; s += stride) {
        int t;
        int64_t b, q0, q1;
        split_slot(s, B, Binv, t, b);
        if (!bag_range(off, s, nnz, q0, q1) && lg == 0) record_bad_offsets(err);
        if (q0 == q1) continue;
        const uint64_t card = (uint64_t)__ldg(p.cards + t);
        const float* grow = gout + (b * p.T + t) * (int64_t)p.d;
        typename V::T gv[KC];
#pragma unroll
        for (int k = 0; k < KC; ++k)
            if (col.v[k]) gv[k] = V::scale(V::ldcs(grow + col.e[k]), scale);
        for (int64_t q = q0; q < q1; ++q) {
            const int64_t id = __ldg(idx + q);
            if ((uint64_t)id >= card) {
                if (lg == 0) record_bad_id(err, q);
                continue;
            }
            const uint64_t kb = hash_key(p, (uint64_t)id, t, 0);
#pragma unroll
            for (int k = 0; k < KC; ++k) {
                if (!col.v[k]) continue;
                const uint64_t x = hash_bucket(p, kb + col.j[k]);
                Acc<VW, AT>::red(target + G * x + col.z[k], gv[k]);
                if (TOUCH && col.z[k] == 0) mark_touched(tc, x);
            }
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
    return a.x != 0.0 || a.y != 0.0 || b.x != 0.0 || b.y != 0.0;
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
        if (g[e] == (GT)0) continue;
        const float gv = to_f32(g[e]);
        if (gv != 0.f) {
            if (ADA) adagrad_elem(w[e], Ga[e], gv, lr, eps);
            else sgd_elem(w[e], gv, lr);
        }
        g[e] = (GT)0;
    }
}

// Gradient export: out[e] = fp32(g[e]) and g[e] = 0, over all of M.
__global__ void __launch_bounds__(kThreads)
k_grad_export(double* __restrict__ g, float* __restrict__ out, int64_t M) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < M; e += stride) {
        const double v = g[e];
        out[e] = to_f32(v);
        if (v != 0.0) g[e] = 0.0;
    }
}

// Touched-block pass: one warp per distinct block start x (from the scatter's
// list).  Element e = x*G + z belongs to the LAST marked start at or below it
// (no marked bucket in (x, x + z/G]), so every element is updated exactly
// once and without atomics even though blocks overlap when G < L.
template <bool ADA, typename GT>
__global__ void __launch_bounds__(kThreads)
k_update_touched(float* __restrict__ w, float* __restrict__ Ga, GT* __restrict__ g,
                 Touched tc, int64_t G, int L, float lr, float eps) {
    const int lane = threadIdx.x & 31;
    unsigned long long n = *tc.count;
    if ((int64_t)n > tc.cap) n = (unsigned long long)tc.cap;
    const int64_t stride = (int64_t)gridDim.x * kWarps;
    for (int64_t it = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5); it < (int64_t)n;
         it += stride) {
        const uint64_t x = (uint64_t)tc.list[it];
        for (int z = lane; z < L; z += 32) {
            const int nb = (int)(z / G);   // following starts that could also cover e
            bool owner = true;
            for (int m0 = 1; m0 <= nb && owner; m0 += 32) {
                const uint64_t y = x + (uint64_t)m0;
                const uint64_t w0 = tc.bitmap[y >> 5];
                const uint64_t w1 = tc.bitmap[(y >> 5) + 1];
                const uint64_t win = ((w1 << 32) | w0) >> (y & 31);
                const int cnt = (nb - m0 + 1) < 32 ? (nb - m0 + 1) : 32;
                const uint64_t mask = (cnt >= 32) ? 0xffffffffull : ((1ull << cnt) - 1);
                if (win & mask) owner = false;
            }
            if (!owner) continue;
            const int64_t e = (int64_t)x * G + z;
            const GT raw = g[e];
            if (raw == (GT)0) continue;
            const float gv = to_f32(raw);
            if (gv != 0.f) {
                if (ADA) adagrad_elem(w[e], Ga[e], gv, lr, eps);
                else sgd_elem(w[e], gv, lr);
            }
            g[e] = (GT)0;
        }
    }
}

__global__ void __launch_bounds__(kThreads) k_touched_clear(Touched tc) {
    unsigned long long n = *tc.count;
    if ((int64_t)n > tc.cap) n = (unsigned long long)tc.cap;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < (int64_t)n; i += stride)
        tc.bitmap[(uint64_t)tc.list[i] >> 5] = 0u;
}

template <int VW, int KC>
cudaError_t forward_inst(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                         const int64_t* off, int64_t B, const float* w, float* out, DevError* err,
                         int sm_count, cudaStream_t st) {
    const int64_t nbags = (int64_t)p.T * B;
    const int64_t per_block = (int64_t)kWarps * (32 >> lay.log2gs);
    const int grid = grid_for(k_forward<VW, KC>, sm_count, (nbags + per_block - 1) / per_block);
    k_forward<VW, KC><<<grid, kThreads, 0, st>>>(p, idx, nnz, off, B, UINT64_MAX / (uint64_t)B, w,
                                                  out, err, lay.log2gs);
    return cudaGetLastError();
}

template <int VW, int KC, bool TOUCH, typename AT>
cudaError_t scatter_inst(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                         const int64_t* off, int64_t B, const float* gout, float scale,
                         AT* target, const Touched& tc, DevError* err, int sm_count,
                         cudaStream_t st) {
    const int64_t nbags = (int64_t)p.T * B;
    const int64_t per_block = (int64_t)kWarps * (32 >> lay.log2gs);
    const int grid = grid_for(k_scatter<VW, KC, TOUCH, AT>, sm_count,
                              (nbags + per_block - 1) / per_block);
    k_scatter<VW, KC, TOUCH, AT><<<grid, kThreads, 0, st>>>(p, idx, nnz, off, B,
                                                            UINT64_MAX / (uint64_t)B, gout, scale,
                                                            target, tc, err, lay.log2gs);
    return cudaGetLastError();
}

template <int VW, int KC, typename AT>
cudaError_t scatter_touch(bool touch, const DevParams& p, const RowLayout& lay,
                          const int64_t* idx, int64_t nnz, const int64_t* off, int64_t B,
                          const float* gout, float scale, AT* target, const Touched* tc,
                          DevError* err, int sm_count, cudaStream_t st) {
    Touched none{};
    if (touch)
        return scatter_inst<VW, KC, true, AT>(p, lay, idx, nnz, off, B, gout, scale, target, *tc,
                                              err, sm_count, st);
    return scatter_inst<VW, KC, false, AT>(p, lay, idx, nnz, off, B, gout, scale, target, none,
                                           err, sm_count, st);
}

template <typename AT>
cudaError_t scatter_dispatch(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                             int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                             float scale, AT* target, const Touched* touched, DevError* err,
                             int sm_count, cudaStream_t st) {
    const bool tch = touched != nullptr;
#define PSS_SC(VW, KC) \
    return scatter_touch<VW, KC, AT>(tch, p, lay, idx, nnz, off, B, grad_out, scale, target, \
                                     touched, err, sm_count, st)
    if (lay.vw == 4) {
        switch (lay.kc) {
            case 1: PSS_SC(4, 1);
            case 2: PSS_SC(4, 2);
            case 4: PSS_SC(4, 4);
        }
    } else {
        switch (lay.kc) {
            case 1: PSS_SC(1, 1);
            case 2: PSS_SC(1, 2);
            case 4: PSS_SC(1, 4);
            case 8: PSS_SC(1, 8);
            case 16: PSS_SC(1, 16);
        }
    }
#undef PSS_SC
    return cudaErrorInvalidValue;
}

template <bool ADA, typename GT>
cudaError_t update_dense_inst(float* w, float* Ga, GT* g, int64_t M, float lr, float eps,
                              int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_update_dense<ADA, GT>, sm_count, ((M >> 2) + kThreads) / kThreads);
    k_update_dense<ADA, GT><<<grid, kThreads, 0, st>>>(w, Ga, g, M, lr, eps);
    return cudaGetLastError();
}

template <bool ADA, typename GT>
cudaError_t update_touched_inst(float* w, float* Ga, GT* g, const Touched& tc, int64_t G,
                                int32_t L, float lr, float eps, int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_update_touched<ADA, GT>, sm_count, (tc.cap + kWarps - 1) / kWarps);
    k_update_touched<ADA, GT><<<grid, kThreads, 0, st>>>(w, Ga, g, tc, G, L, lr, eps);
    return cudaGetLastError();
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
    k_locations<<<grid, kThreads, 0, st>>>(p, idx, nnz, off, B, UINT64_MAX / (uint64_t)B, locs, err);
    return cudaGetLastError();
}

cudaError_t launch_forward(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* w, float* out,
                           DevError* err, int sm_count, cudaStream_t st) {
    if (lay.vw == 4) {
        switch (lay.kc) {
            case 1: return forward_inst<4, 1>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 2: return forward_inst<4, 2>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 4: return forward_inst<4, 4>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
        }
    } else {
        switch (lay.kc) {
            case 1: return forward_inst<1, 1>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 2: return forward_inst<1, 2>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 4: return forward_inst<1, 4>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 8: return forward_inst<1, 8>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
            case 16: return forward_inst<1, 16>(p, lay, idx, nnz, off, B, w, out, err, sm_count, st);
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_scatter(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                           float scale, float* target, const Touched* touched, DevError* err,
                           int sm_count, cudaStream_t st) {
    return scatter_dispatch<float>(p, lay, idx, nnz, off, B, grad_out, scale, target, touched, err,
                                   sm_count, st);
}

cudaError_t launch_scatter64(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                             int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                             double* target, const Touched* touched, DevError* err, int sm_count,
                             cudaStream_t st) {
    return scatter_dispatch<double>(p, lay, idx, nnz, off, B, grad_out, 1.0f, target, touched,
                                    err, sm_count, st);
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
    k_grad_export<<<grid, kThreads, 0, st>>>(g, out, M);
    return cudaGetLastError();
}

cudaError_t launch_touched_clear(const Touched& tc, int sm_count, cudaStream_t st) {
    const int grid = grid_for(k_touched_clear, sm_count, (tc.cap + kThreads - 1) / kThreads);
    k_touched_clear<<<grid, kThreads, 0, st>>>(tc);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return cudaMemsetAsync(tc.count, 0, sizeof(unsigned long long), st);
}

}  // namespace pss
