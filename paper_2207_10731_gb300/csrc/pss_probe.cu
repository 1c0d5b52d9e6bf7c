// Measurement kernels of the L2 roofline: the rates at which this GPU serves
// the two kinds of L2 traffic the method makes when the shared array fits in
// L2 -- random gathers of 128-byte blocks (the forward's block reads) and
// reductions into random addresses (the dense branch of Algorithm 1: fp64
// scalar and 16-byte fp32 vector reductions).  They do no method arithmetic;
// bench.py times them with CUDA events to get the L2 peaks it reports beside
// the measured HBM copy peak.
#include <cstdint>

#include "pss.h"
#include "pss_device.cuh"
#include "pss_internal.h"

using namespace pss;

namespace {

constexpr int kPU = 8;   // independent accesses in flight per lane

// Index streams that cost a few instructions per access, so that the probes
// measure the memory system rather than their own arithmetic: a 32-bit
// linear congruential step (Knuth's MMIX multiplier truncated to 32 bits)
// whose top bits select one of `mask + 1` blocks (a power of two).
__device__ __forceinline__ uint32_t lcg_next(uint32_t s) { return s * 1664525u + 1013904223u; }

// Gather: each warp reads `iters` random 128-byte blocks (lane l reads word l).
__global__ void __launch_bounds__(kThreads)
k_probe_gather(const float* __restrict__ buf, uint32_t mask, int log2n, int iters,
               float* __restrict__ out) {
    pdl_prologue();
    const int lane = threadIdx.x & 31;
    uint32_t st = (uint32_t)(blockIdx.x * kWarps + (threadIdx.x >> 5)) * 2654435761u + 12345u;
    float acc = 0.f;
    for (int k0 = 0; k0 < iters; k0 += kPU) {
        float v[kPU];
#pragma unroll
        for (int u = 0; u < kPU; ++u) {
            st = lcg_next(st);
            const uint32_t b = (st >> (32 - log2n)) & mask;
            v[u] = __ldcg(buf + (size_t)b * 32 + lane);
        }
#pragma unroll
        for (int u = 0; u < kPU; ++u) acc += v[u];
    }
    if (acc == 1.2345f) out[0] = acc;   // keeps the loads
}

// Streaming read: in round k, warp w reads line (k * warps + w) mod lines.
__global__ void __launch_bounds__(kThreads)
k_probe_stream(const float* __restrict__ buf, uint32_t nlines, int iters, float* __restrict__ out) {
    pdl_prologue();
    const int lane = threadIdx.x & 31;
    const uint32_t nw = gridDim.x * kWarps;
    uint32_t line = (blockIdx.x * kWarps + (threadIdx.x >> 5)) % nlines;
    float acc = 0.f;
    for (int k0 = 0; k0 < iters; k0 += kPU) {
        float v[kPU];
#pragma unroll
        for (int u = 0; u < kPU; ++u) {
            v[u] = __ldcg(buf + (size_t)line * 32 + lane);
            line += nw;
            while (line >= nlines) line -= nlines;
        }
#pragma unroll
        for (int u = 0; u < kPU; ++u) acc += v[u];
    }
    if (acc == 1.2345f) out[0] = acc;   // keeps the loads
}

// Reductions, as the method's kernels issue them: each warp adds into `iters`
// random blocks, its lanes on consecutive elements -- 32 doubles (256 bytes,
// red.global.add.f64) or 32 16-byte fp32 vectors (512 bytes,
// red.global.add.v4.f32) per instruction, among `mask + 1` blocks.
template <bool V4>
__global__ void __launch_bounds__(kThreads)
k_probe_red(void* __restrict__ buf, uint32_t mask, int log2n, int iters) {
    pdl_prologue();
    const int lane = threadIdx.x & 31;
    uint32_t st = (uint32_t)(blockIdx.x * kWarps + (threadIdx.x >> 5)) * 2654435761u + 12345u;
    for (int k = 0; k < iters; ++k) {
        st = lcg_next(st);
        const size_t i = (size_t)((st >> (32 - log2n)) & mask) * 32 + lane;
        if (V4)
            red_add_v4(static_cast<float*>(buf) + 4 * i, make_float4(1.f, 1.f, 1.f, 1.f));
        else
            red_add_f64(static_cast<double*>(buf) + i, 1.0);
    }
}

int floor_log2(int64_t v) {
    int l = 0;
    while ((int64_t(1) << (l + 1)) <= v) ++l;
    return l;
}

}  // namespace

extern "C" pss_status pss_probe_l2(int32_t kind, void* buf, int64_t bytes, int64_t iters,
                                   int32_t ctas, pss_stream stream) {
    if (kind < 0 || kind > 3 || !buf || bytes < 4096 || iters <= 0 || iters > (1 << 24) ||
        ctas <= 0)
        return PSS_ERR_INVALID_ARG;
    if (((uintptr_t)buf & 255u) != 0) return PSS_ERR_INVALID_ARG;
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, buf) != cudaSuccess || a.type != cudaMemoryTypeDevice) {
        cudaGetLastError();
        return PSS_ERR_INVALID_ARG;
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e;
    // the last 128 bytes of the buffer hold the (never taken) keep-alive store
    const int64_t lines = (bytes - 128) / 128;
    const int it = (int)(((iters + kPU - 1) / kPU) * kPU);
    if (kind == 0 || kind == 3) {
        float* keep = reinterpret_cast<float*>(static_cast<char*>(buf) + bytes - 4);
        const int lg = floor_log2(lines);   // the gather uses 2^lg of the lines
        if (kind == 0)
            e = launch_k(k_probe_gather, dim3(ctas), dim3(kThreads), 0, st,
                         static_cast<const float*>(buf), (uint32_t)((int64_t(1) << lg) - 1), lg,
                         it, keep);
        else
            e = launch_k(k_probe_stream, dim3(ctas), dim3(kThreads), 0, st,
                         static_cast<const float*>(buf),
                         (uint32_t)(lines < 0xffffffffLL ? lines : 0xffffffffLL), it, keep);
    } else {
        const int64_t n = bytes / (kind == 1 ? 256 : 512);   // blocks of 32 lanes' elements
        const int lg = floor_log2(n < 0xffffffffLL ? n : 0xffffffffLL);
        const uint32_t mask = (uint32_t)((int64_t(1) << lg) - 1);
        e = (kind == 1) ? launch_k(k_probe_red<false>, dim3(ctas), dim3(kThreads), 0, st, buf, mask,
                                   lg, (int)iters)
                        : launch_k(k_probe_red<true>, dim3(ctas), dim3(kThreads), 0, st, buf, mask,
                                   lg, (int)iters);
    }
    return e == cudaSuccess ? PSS_OK : PSS_ERR_CUDA;
}
