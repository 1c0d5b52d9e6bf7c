// Device helpers of libpss: the location hash and small memory primitives.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "pss_internal.h"

namespace pss {

constexpr uint64_t kP61 = (uint64_t(1) << 61) - 1;

// Bucket of one hashed key (universal hashing of Sec. 2.5, in the fixed form
// documented in pss.h):  x = ((A*key + B0) mod (2^61-1)) mod R.
// A*key < 2^122 is folded with 2^61 == 1 (mod P); "mod R" uses the
// precomputed Rinv = floor((2^64-1)/R): q' = umulhi(s, Rinv) is q or q-1 for
// s < 2^64 (Barrett, CRYPTO '86), so one conditional subtraction is exact.
__device__ __forceinline__ uint64_t affine_mod_p61(uint64_t a, uint64_t key, uint64_t b) {
    const uint64_t lo = a * key;
    const uint64_t hi = __umul64hi(a, key);               // < 2^58
    uint64_t s = (lo & kP61) + ((lo >> 61) | (hi << 3));  // < 2^62
    s += b;                                               // < 2^62 + 2^61
    s = (s & kP61) + (s >> 61);                           // < 2^61 + 3
    return (s >= kP61) ? s - kP61 : s;
}

__device__ __forceinline__ uint64_t hash_bucket(const DevParams& p, uint64_t key) {
    const uint64_t s = affine_mod_p61(p.A, key, p.B0);
    const uint64_t q = __umul64hi(s, p.Rinv);
    uint64_t r = s - q * p.R;
    return (r >= p.R) ? r - p.R : r;
}

__device__ __forceinline__ uint64_t hash_key(const DevParams& p, uint64_t id, int t, int j) {
    return (id * (uint64_t)p.T + (uint64_t)t) * (uint64_t)p.J + (uint64_t)j;
}

// Signed hashing: the sign s = -1 of a key whose sign hash (A2*key + B2) mod
// (2^61-1) is odd, as the fp32 sign bit (0x80000000); 0 for s = +1 and
// whenever signed hashing is off (smask == 0).  Bucket indices carry it in
// their bit 31 (R < 2^31 with signed hashing), which is where fp32 keeps its
// sign, so a value is signed by an XOR with the index's masked bit.
__device__ __forceinline__ uint32_t hash_sign_bit(const DevParams& p, uint64_t key) {
    if (!p.smask) return 0u;
    return (uint32_t)(affine_mod_p61(p.A2, key, p.B2) & 1u) << 31;
}

__device__ __forceinline__ float sign_by(float v, uint32_t sbit) {
    return __uint_as_float(__float_as_uint(v) ^ sbit);
}
__device__ __forceinline__ float4 sign_by(float4 v, uint32_t sbit) {
    return make_float4(sign_by(v.x, sbit), sign_by(v.y, sbit), sign_by(v.z, sbit),
                       sign_by(v.w, sbit));
}

__device__ __forceinline__ void record_bad_id(DevError* err, int64_t q) {
    atomicMin(&err->first_bad, (unsigned long long)q);
}

__device__ __forceinline__ void record_bad_offsets(DevError* err) {
    atomicOr(&err->flags, kErrOffsets);
}

// 16-byte vector reduction into global memory (sm_90+), relaxed, no return.
__device__ __forceinline__ void red_add_v4(float* addr, float4 v) {
    asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};"
                 :: "l"(addr), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w) : "memory");
}

__device__ __forceinline__ void red_add_f64(double* addr, double v) {
    asm volatile("red.global.add.f64 [%0], %1;" :: "l"(addr), "d"(v) : "memory");
}

__device__ __forceinline__ void red_add_f32(float* addr, float v) {
    asm volatile("red.global.add.f32 [%0], %1;" :: "l"(addr), "f"(v) : "memory");
}

// Compensated (Kahan) accumulation: error independent of the bag length.
__device__ __forceinline__ void kahan_add(float& s, float& c, float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
}

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// Programmatic dependent launch.  Every kernel of the library starts with
// pdl_prologue(), which waits until the previous kernel on the stream has
// completed and its memory is visible (a no-op when the previous work was not
// a kernel launched this way), before any global access.  So a kernel never
// overlaps the one before it in anything it reads or writes; only the launch
// latency between them is hidden.
__device__ __forceinline__ void pdl_prologue() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launch with programmatic stream serialization (see pdl_prologue).
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

inline int ceil_log2(int v) {
    int l = 0;
    while ((1 << l) < v) ++l;
    return l;
}

// Grid of a grid-stride kernel: all CTAs that fit at once, capped by the work.
template <typename K>
int grid_for(K kernel, int sm_count, int64_t work_blocks, size_t smem = 0) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, smem) !=
            cudaSuccess ||
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

// Exact fp32 -> fp64 widening from the IEEE-754 fields, in integer
// arithmetic only (the FP64 pipe of this part is slow, and a conversion left
// in a predicated branch would still occupy it): the exponent is re-biased
// (127 -> 1023) and the 23-bit fraction moved to the top of the 52-bit one; a
// subnormal input is normalised at its leading one; zeros, infinities and NaNs
// keep their sign and fraction.
__device__ __forceinline__ double widen(float f) {
    const uint32_t u = __float_as_uint(f);
    const uint64_t sign = (uint64_t)(u & 0x80000000u) << 32;
    const uint32_t e = (u >> 23) & 0xffu;
    const uint32_t m = u & 0x7fffffu;
    uint64_t bits;
    if (e == 0xffu) {
        bits = sign | (uint64_t(0x7ff) << 52) | ((uint64_t)m << 29);
    } else if (e != 0u) {
        bits = sign | ((uint64_t)(e + 896u) << 52) | ((uint64_t)m << 29);
    } else if (m == 0u) {
        bits = sign;
    } else {
        // m * 2^-149 with the leading one at bit p: exponent p - 149
        const int p = 31 - __clz(m);
        bits = sign | ((uint64_t)(p + 874) << 52) |
               (((uint64_t)m << (52 - p)) & ((uint64_t(1) << 52) - 1));
    }
    return __longlong_as_double((long long)bits);
}

// Reduction of one VW-wide column into an fp32 or fp64 accumulator.
template <int VW, typename AT>
struct Acc;
template <int VW>
struct Acc<VW, float> {
    static __device__ __forceinline__ void red(float* p, typename Vec<VW>::T v) { Vec<VW>::red(p, v); }
};
template <>
struct Acc<1, double> {
    static __device__ __forceinline__ void red(double* p, float v) { red_add_f64(p, widen(v)); }
};

// fp64 -> fp32, rounded to nearest (ties to even), in integer arithmetic
// only (the FP64 pipe of this part is slow).  The 53-bit significand is cut
// to 24 bits (or, below the normal range, to units of 2^-149) and rounded on
// the dropped bits; a carry out of the fraction moves into the exponent,
// which is also how rounding reaches the next binade or infinity.
__device__ __forceinline__ float narrow(double v) {
    const uint64_t b = (uint64_t)__double_as_longlong(v);
    const uint32_t sign = (uint32_t)(b >> 32) & 0x80000000u;
    const int e = (int)((b >> 52) & 0x7ff);
    const uint64_t m = b & ((uint64_t(1) << 52) - 1);
    if (e == 0x7ff)   // infinity, or NaN (kept quiet, top fraction bits kept)
        return __uint_as_float(sign | 0x7f800000u | (m ? (0x400000u | (uint32_t)(m >> 29)) : 0u));
    const int ef = e - 1023 + 127;
    if (ef >= 0xff) return __uint_as_float(sign | 0x7f800000u);
    if (ef >= 1) {
        const uint32_t mm = (uint32_t)(m >> 29);
        const uint64_t rem = m & ((uint64_t(1) << 29) - 1);
        const uint64_t half = uint64_t(1) << 28;
        uint32_t r = ((uint32_t)ef << 23) | mm;
        if (rem > half || (rem == half && (mm & 1u))) r += 1u;
        return __uint_as_float(sign | r);
    }
    if (e == 0) return __uint_as_float(sign);   // below 2^-1022: rounds to zero
    // significand S = 2^52 + m; the value in units of 2^-149 is S / 2^sh
    const int sh = 926 - e;                      // >= 30 here
    if (sh > 54) return __uint_as_float(sign);
    const uint64_t S = (uint64_t(1) << 52) | m;
    uint32_t q = (uint32_t)(S >> sh);
    const uint64_t rem = S & ((uint64_t(1) << sh) - 1);
    const uint64_t half = uint64_t(1) << (sh - 1);
    if (rem > half || (rem == half && (q & 1u))) q += 1u;
    return __uint_as_float(sign | q);
}

// Accumulator element -> fp32 gradient (rounded once, to nearest).
__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(double v) { return narrow(v); }

// Non-zero test (+0 and -0 are zero), fp64 by its bits.
__device__ __forceinline__ bool nonzero(float v) { return v != 0.f; }
__device__ __forceinline__ bool nonzero(double v) {
    return ((uint64_t)__double_as_longlong(v) << 1) != 0u;
}

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


// Record distinct block starts in the touched bitmap / list: the lane that
// sets a bucket's bit first appends it; the appends of a warp share one
// atomic on the list counter.  All 32 lanes must call this together.
__device__ __forceinline__ void mark_touched_warp(const Touched& tc, uint64_t x, bool valid,
                                                  int lane) {
    bool first = false;
    if (valid) {
        uint32_t* wp = tc.bitmap + (x >> 5);
        const uint32_t bit = 1u << (x & 31);
        if (!(*reinterpret_cast<volatile uint32_t*>(wp) & bit)) first = !(atomicOr(wp, bit) & bit);
    }
    const unsigned m = __ballot_sync(0xffffffffu, first);
    if (m == 0u) return;
    const int leader = __ffs(m) - 1;
    unsigned long long base = 0;
    if (lane == leader) base = atomicAdd(tc.count, (unsigned long long)__popc(m));
    base = __shfl_sync(0xffffffffu, base, leader);
    if (first) {
        const unsigned long long slot = base + (unsigned long long)__popc(m & ((1u << lane) - 1u));
        if ((int64_t)slot < tc.cap) tc.list[slot] = (int64_t)x;
    }
}

}  // namespace pss
