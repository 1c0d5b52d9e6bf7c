// Sorted backward path (the sparse branch of Algorithm 1: find the distinct
// locations, sum the contributions of each, then apply them).
//
// Input, written by the forward pass of the same batch:
//   pair_x[p]  bucket x of pair p = q*J + j (block start G*x), or 0xffffffff
//              for an id outside its table;
//   q_row[q]   output row b*T + t of the bag that holds id q;
//   cnt[x]     number of valid pairs with bucket x (the forward zeroes and
//              fills it while it hashes).
// Steps (all on the caller's stream):
//   1. scan     start[x] = sum of cnt[y] for y < x (three kernels);
//               statistics: valid pairs and distinct buckets;
//   2. scatter  each pair takes slot start[x] + (--cnt[x]) of sorted_e, which
//               holds (x, r = row*J + j): the bucket and the upstream-gradient
//               chunk to add;
//   3. reduce   the sorted entries are cut into tasks of kPiece consecutive
//               entries; one group of lanes per task owns 16-byte columns of
//               the block, adds the chunks of each run of equal x with
//               compensated (Kahan) fp32 sums, and adds every run's sum once
//               into the fp64 gradient accumulator g[G*x + z] -- one reduction
//               per run and element instead of one per contribution, and no
//               queue of reductions on a hot address.
// The optimizer pass over g follows (pss_kernels.cu).
#include <climits>

#include "pss_device.cuh"
#include "pss_internal.h"

namespace pss {
namespace {

constexpr uint32_t kBad = 0xffffffffu;
constexpr int kScanThreads = 1024;
constexpr int kScanPerThread = 8;
constexpr int kScanChunk = kScanThreads * kScanPerThread;
constexpr int kRU = 4;            // entries in flight per group

// Block-wide exclusive scan of one value per thread (kScanThreads threads).
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* s_warp,
                                                         uint32_t* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const uint32_t w = (lane < (kScanThreads >> 5)) ? s_warp[lane] : 0u;
        uint32_t ws = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, ws, o);
            if (lane >= o) ws += y;
        }
        if (lane < (kScanThreads >> 5)) s_warp[lane] = ws - w;
        if (lane == 31) s_warp[32] = ws;
    }
    __syncthreads();
    const uint32_t r = s_warp[warp] + x - v;
    *total = s_warp[32];
    __syncthreads();
    return r;
}

// Per chunk of kScanChunk counters: entries and non-empty buckets.
__global__ void __launch_bounds__(kScanThreads)
k_scan_reduce(const uint32_t* __restrict__ cnt, int64_t R, uint32_t* __restrict__ bsum,
              uint32_t* __restrict__ bnz) {
    __shared__ uint32_t s_warp[33];
    const int64_t base = (int64_t)blockIdx.x * kScanChunk;
    uint32_t sum = 0, nz = 0;
#pragma unroll
    for (int i = 0; i < kScanPerThread; ++i) {
        const int64_t e = base + (int64_t)i * kScanThreads + threadIdx.x;
        const uint32_t c = (e < R) ? cnt[e] : 0u;
        sum += c;
        nz += (c != 0u);
    }
    uint32_t tot;
    block_exclusive_scan(sum, s_warp, &tot);
    if (threadIdx.x == 0) bsum[blockIdx.x] = tot;
    block_exclusive_scan(nz, s_warp, &tot);
    if (threadIdx.x == 0) bnz[blockIdx.x] = tot;
}

// Exclusive scan of the chunk sums (one block).  stats[0] = valid pairs,
// stats[1] = distinct buckets.
// Exclusive scans of the chunk sums and of the chunk non-empty counts (one
// block).  stats[0] = valid pairs, stats[1] = distinct buckets, which is also
// the length of the touched list when one is built.
__global__ void __launch_bounds__(kScanThreads)
k_scan_top(uint32_t* __restrict__ bsum, uint32_t* __restrict__ bnz, int64_t nblk,
           unsigned long long* __restrict__ stats, unsigned long long* __restrict__ touched_count) {
    __shared__ uint32_t s_warp[33];
    __shared__ uint32_t s_carry[2];
    if (threadIdx.x < 2) s_carry[threadIdx.x] = 0;
    __syncthreads();
    for (int64_t b0 = 0; b0 < nblk; b0 += kScanThreads) {
        const int64_t b = b0 + threadIdx.x;
        const bool in = b < nblk;
        const uint32_t v = in ? bsum[b] : 0u;
        const uint32_t z = in ? bnz[b] : 0u;
        uint32_t tot_v, tot_z;
        const uint32_t ex_v = block_exclusive_scan(v, s_warp, &tot_v);
        const uint32_t ex_z = block_exclusive_scan(z, s_warp, &tot_z);
        const uint32_t cv = s_carry[0], cz = s_carry[1];
        if (in) {
            bsum[b] = cv + ex_v;
            bnz[b] = cz + ex_z;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            s_carry[0] = cv + tot_v;
            s_carry[1] = cz + tot_z;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        stats[0] = s_carry[0];
        stats[1] = s_carry[1];
        if (touched_count) *touched_count = s_carry[1];
    }
}

// start[x] = exclusive prefix of cnt; start[R] = total.  With a touched
// list, the non-empty buckets are listed in order and their bits set.
__global__ void __launch_bounds__(kScanThreads)
k_scan_apply(const uint32_t* __restrict__ cnt, int64_t R, const uint32_t* __restrict__ bsum,
             const uint32_t* __restrict__ bnz, uint32_t* __restrict__ start, Touched tc) {
    __shared__ uint32_t s_warp[33];
    const int64_t base = (int64_t)blockIdx.x * kScanChunk;
    uint32_t c[kScanPerThread];
    uint32_t sum = 0, nz = 0;
#pragma unroll
    for (int i = 0; i < kScanPerThread; ++i) {
        const int64_t e = base + (int64_t)threadIdx.x * kScanPerThread + i;
        c[i] = (e < R) ? cnt[e] : 0u;
        sum += c[i];
        nz += (c[i] != 0u);
    }
    uint32_t tot;
    uint32_t run = bsum[blockIdx.x] + block_exclusive_scan(sum, s_warp, &tot);
    uint32_t zrun = bnz[blockIdx.x] + block_exclusive_scan(nz, s_warp, &tot);
#pragma unroll
    for (int i = 0; i < kScanPerThread; ++i) {
        const int64_t e = base + (int64_t)threadIdx.x * kScanPerThread + i;
        if (e < R) start[e] = run;
        run += c[i];
        if (e == R - 1) start[R] = run;
        if (tc.list && c[i] != 0u) {
            if ((int64_t)zrun < tc.cap) tc.list[zrun] = e;
            atomicOr(tc.bitmap + (e >> 5), 1u << (e & 31));
            ++zrun;
        }
    }
}

// Slot of every valid pair; cnt counts back down to zero.  Lanes of a warp
// with the same bucket share one atomic (the leader takes n slots at once);
// each warp keeps kSU such rounds in flight.
constexpr int kSU = 4;

__global__ void __launch_bounds__(kThreads)
k_sort_scatter(const uint32_t* __restrict__ pair_x, int64_t npairs, const uint32_t* __restrict__ q_row,
               int J, int log2J, const uint32_t* __restrict__ start, uint32_t* __restrict__ cnt,
               unsigned long long* __restrict__ sorted_e) {
    const int lane = threadIdx.x & 31;
    const int64_t wstride = (int64_t)gridDim.x * blockDim.x * kSU;
    for (int64_t p0 = ((int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31)) * kSU; p0 < npairs;
         p0 += wstride) {
        uint32_t x[kSU], row[kSU], st0[kSU], old[kSU], jj[kSU];
        unsigned peers[kSU];
#pragma unroll
        for (int u = 0; u < kSU; ++u) {
            const int64_t p = p0 + u * 32 + lane;
            x[u] = (p < npairs) ? __ldg(pair_x + p) : kBad;
        }
        // loads that do not depend on the slot go first, so they overlap the atomics
#pragma unroll
        for (int u = 0; u < kSU; ++u) {
            const uint32_t pp = (uint32_t)(p0 + u * 32 + lane);   // npairs < 2^32 on this path
            const uint32_t q = (log2J >= 0) ? (pp >> log2J) : pp / (uint32_t)J;
            jj[u] = pp - q * (uint32_t)J;
            row[u] = 0;
            st0[u] = 0;
            if (x[u] != kBad) {
                row[u] = __ldg(q_row + q);
                st0[u] = __ldg(start + x[u]);
            }
        }
#pragma unroll
        for (int u = 0; u < kSU; ++u) {
            peers[u] = __match_any_sync(0xffffffffu, x[u]);
            old[u] = 0;
            if (x[u] != kBad && lane == __ffs(peers[u]) - 1)
                old[u] = atomicSub(cnt + x[u], (uint32_t)__popc(peers[u]));
        }
#pragma unroll
        for (int u = 0; u < kSU; ++u) {
            const int leader = __ffs(peers[u]) - 1;
            const uint32_t o = __shfl_sync(0xffffffffu, old[u], leader);
            if (x[u] == kBad) continue;
            const uint32_t rank = (uint32_t)__popc(peers[u] & ((1u << lane) - 1u));
            const uint32_t slot = st0[u] + o - 1u - rank;
            sorted_e[slot] = ((unsigned long long)x[u] << 32) | (row[u] * (uint32_t)J + jj[u]);
        }
    }
}

// Exact fp32 -> fp64 widening from the IEEE-754 fields (integer pipe): the
// exponent is re-biased (127 -> 1023) and the 23-bit fraction moved to the top
// of the 52-bit one.  Zeros, subnormals, infinities and NaNs take the
// hardware conversion.
__device__ __forceinline__ double widen(float f) {
    const uint32_t u = __float_as_uint(f);
    const uint32_t e = (u >> 23) & 0xffu;
    if (e == 0u || e == 0xffu) return (double)f;
    const uint64_t bits = ((uint64_t)(u & 0x80000000u) << 32) |
                          ((uint64_t)(e + 896u) << 52) | ((uint64_t)(u & 0x7fffffu) << 29);
    return __longlong_as_double((long long)bits);
}

// Reduce: one group of gs lanes per task of kPiece sorted entries; lane lg
// owns columns lg + k*gs of VW elements of the L-element block.  Each run of
// equal x is summed with compensation (Kahan) and added once into the fp64
// accumulator through a shared-memory transpose (so that every fp64
// reduction instruction covers consecutive elements).
constexpr int64_t kPiece = 64;    // sorted entries per reduce task

template <int VW, int KC, bool JPOW2>
__global__ void __launch_bounds__(kThreads, (KC == 1) ? 4 : 1)
k_range_reduce(const unsigned long long* __restrict__ sorted_e,
               const unsigned long long* __restrict__ stats, int64_t npairs,
               const float* __restrict__ gout, int d, int Z, int J, int log2J, int L, int64_t G,
               double* __restrict__ g, Touched tc, int log2gs) {
    using V = Vec<VW>;
    using VT = typename V::T;
    extern __shared__ __align__(16) float s_stage[];   // [groups per CTA][L]
    const int64_t total = (int64_t)(stats[0] < (unsigned long long)npairs ? stats[0] : npairs);
    const int64_t ntasks = (total + kPiece - 1) / kPiece;
    const int lane = threadIdx.x & 31;
    const int gs = 1 << log2gs;
    const int lg = lane & (gs - 1);
    const int gpw = 32 >> log2gs;
    const int grp = (threadIdx.x >> 5) * gpw + (lane >> log2gs);
    float* stage = s_stage + grp * L;
    const unsigned gmask = (gs == 32) ? 0xffffffffu
                                      : (((1u << gs) - 1u) << ((lane >> log2gs) << log2gs));
    const int64_t gstride = (int64_t)gridDim.x * kWarps * gpw;
    float s[KC][VW], c[KC][VW];

    auto flush = [&](uint32_t x) {
#pragma unroll
        for (int k = 0; k < KC; ++k) {
            const int col = (lg + k * gs) * VW;
#pragma unroll
            for (int i = 0; i < VW; ++i) {
                if (col + i < L) stage[col + i] = s[k][i];
                s[k][i] = c[k][i] = 0.f;
            }
        }
        __syncwarp(gmask);
        double* base = g + (int64_t)x * G;
        for (int z = lg; z < L; z += gs) {
            const float val = stage[z];
            if (val != 0.f) red_add_f64(base + z, widen(val));
        }
        __syncwarp(gmask);
    };

    for (int64_t t = (int64_t)blockIdx.x * kWarps * gpw + grp; t < ntasks; t += gstride) {
        const int64_t e0 = t * kPiece;
        const int64_t e1 = (e0 + kPiece < total) ? e0 + kPiece : total;
#pragma unroll
        for (int k = 0; k < KC; ++k)
#pragma unroll
            for (int i = 0; i < VW; ++i) s[k][i] = c[k][i] = 0.f;
        constexpr unsigned long long kNone = (unsigned long long)kBad << 32;
        // entries of the next block are loaded one block ahead
        unsigned long long nxt[kRU];
#pragma unroll
        for (int u = 0; u < kRU; ++u) nxt[u] = (e0 + u < e1) ? __ldg(sorted_e + e0 + u) : kNone;
        uint32_t cur = (uint32_t)(nxt[0] >> 32);
        for (int64_t e = e0; e < e1; e += kRU) {
            uint32_t xs[kRU];
            VT v[kRU][KC];
            unsigned long long ent[kRU];
#pragma unroll
            for (int u = 0; u < kRU; ++u) {
                ent[u] = nxt[u];
                const int64_t en = e + kRU + u;
                nxt[u] = (en < e1) ? __ldg(sorted_e + en) : kNone;
            }
#pragma unroll
            for (int u = 0; u < kRU; ++u) {
                xs[u] = (uint32_t)(ent[u] >> 32);
#pragma unroll
                for (int k = 0; k < KC; ++k)
#pragma unroll
                    for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                if (xs[u] != kBad) {
                    const uint32_t r = (uint32_t)ent[u];
                    const uint32_t row = JPOW2 ? (r >> log2J) : r / (uint32_t)J;
                    const int j = (int)(r - row * (uint32_t)J);
                    const int Lj = (d - j * Z) < Z ? (d - j * Z) : Z;
                    const float* src = gout + (int64_t)row * d + j * Z;
#pragma unroll
                    for (int k = 0; k < KC; ++k) {
                        const int col = (lg + k * gs) * VW;
                        if (col < Lj) v[u][k] = V::ldcs(src + col);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < kRU; ++u) {
                if (xs[u] == kBad) break;
                if (xs[u] != cur) {
                    flush(cur);
                    cur = xs[u];
                }
#pragma unroll
                for (int k = 0; k < KC; ++k)
#pragma unroll
                    for (int i = 0; i < VW; ++i) kahan_add(s[k][i], c[k][i], V::get(v[u][k], i));
            }
        }
        flush(cur);
    }
}

template <int VW, int KC>
cudaError_t reduce_inst(const SortedBuffers& sb, int64_t npairs, const float* gout,
                        const DevParams& p, double* g, const Touched& tc, int log2gs,
                        int sm_count, cudaStream_t st) {
    const int log2J = (p.J & (p.J - 1)) == 0 ? ceil_log2(p.J) : -1;
    const int gpc = kWarps * (32 >> log2gs);
    const size_t smem = sizeof(float) * (size_t)gpc * (size_t)p.L;
    const int64_t ntasks = (npairs + kPiece - 1) / kPiece;   // upper bound
    const int64_t work_blocks = (ntasks + gpc - 1) / gpc;
    if (log2J >= 0) {
        const int grid = grid_for(k_range_reduce<VW, KC, true>, sm_count, work_blocks, smem);
        k_range_reduce<VW, KC, true><<<grid, kThreads, smem, st>>>(
            sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, log2J, p.L, p.G, g, tc, log2gs);
    } else {
        const int grid = grid_for(k_range_reduce<VW, KC, false>, sm_count, work_blocks, smem);
        k_range_reduce<VW, KC, false><<<grid, kThreads, smem, st>>>(
            sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, 0, p.L, p.G, g, tc, log2gs);
    }
    return cudaGetLastError();
}

}  // namespace

int64_t sorted_scan_blocks(int64_t R) { return (R + kScanChunk - 1) / kScanChunk; }



cudaError_t launch_sorted_scan(const SortedBuffers& sb, int64_t R, const Touched* touched,
                               cudaStream_t st) {
    const int64_t nblk = sorted_scan_blocks(R);
    const Touched tc = touched ? *touched : Touched{};
    k_scan_reduce<<<(unsigned)nblk, kScanThreads, 0, st>>>(sb.cnt, R, sb.bsum, sb.bnz);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_scan_top<<<1, kScanThreads, 0, st>>>(sb.bsum, sb.bnz, nblk, sb.stats, tc.count);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_scan_apply<<<(unsigned)nblk, kScanThreads, 0, st>>>(sb.cnt, R, sb.bsum, sb.bnz, sb.start, tc);
    return cudaGetLastError();
}

cudaError_t launch_sorted_scatter(const SortedBuffers& sb, int64_t npairs, int J, int sm_count,
                                  cudaStream_t st) {
    const int log2J = (J & (J - 1)) == 0 ? ceil_log2(J) : -1;
    const int grid = grid_for(k_sort_scatter, sm_count, (npairs + kThreads - 1) / kThreads);
    k_sort_scatter<<<grid, kThreads, 0, st>>>(sb.pair_x, npairs, sb.q_row, J, log2J, sb.start,
                                              sb.cnt, sb.sorted_e);
    return cudaGetLastError();
}

cudaError_t launch_sorted_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, double* g, const Touched* touched,
                                 int sm_count, cudaStream_t st) {
    const Touched tc = touched ? *touched : Touched{};
    const bool vec = (p.Z % 4 == 0) && (p.d % 4 == 0) && (((uintptr_t)gout & 15u) == 0);
    const int vw = vec ? 4 : 1;
    const int V = (p.L + vw - 1) / vw;
    const int log2gs = V <= 32 ? ceil_log2(V) : 5;
    const int kc = V <= 32 ? 1 : (1 << ceil_log2((V + 31) / 32));
#define PSS_RD(VW, KC) return reduce_inst<VW, KC>(sb, npairs, gout, p, g, tc, log2gs, sm_count, st)
    if (vec) {
        switch (kc) {
            case 1: PSS_RD(4, 1);
            case 2: PSS_RD(4, 2);
            case 4: PSS_RD(4, 4);
        }
    } else {
        switch (kc) {
            case 1: PSS_RD(1, 1);
            case 2: PSS_RD(1, 2);
            case 4: PSS_RD(1, 4);
            case 8: PSS_RD(1, 8);
            case 16: PSS_RD(1, 16);
        }
    }
#undef PSS_RD
    return cudaErrorInvalidValue;
}

}  // namespace pss
