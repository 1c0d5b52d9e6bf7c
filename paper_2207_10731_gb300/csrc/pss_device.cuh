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
__device__ __forceinline__ uint64_t hash_bucket(const DevParams& p, uint64_t key) {
    const uint64_t lo = p.A * key;
    const uint64_t hi = __umul64hi(p.A, key);            // < 2^58
    uint64_t s = (lo & kP61) + ((lo >> 61) | (hi << 3));  // < 2^62
    s += p.B0;                                            // < 2^62 + 2^61
    s = (s & kP61) + (s >> 61);                           // < 2^61 + 3
    s = (s >= kP61) ? s - kP61 : s;
    const uint64_t q = __umul64hi(s, p.Rinv);
    uint64_t r = s - q * p.R;
    return (r >= p.R) ? r - p.R : r;
}

__device__ __forceinline__ uint64_t hash_key(const DevParams& p, uint64_t id, int t, int j) {
    return (id * (uint64_t)p.T + (uint64_t)t) * (uint64_t)p.J + (uint64_t)j;
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

}  // namespace pss
