// Sorted backward path (the sparse branch of Algorithm 1: find the distinct
// locations, sum the contributions of each, then apply them).
//
// Input, written by the forward pass of the same batch:
//   pair_x[p]  bucket x of pair p = q*J + j (block start G*x), or 0xffffffff
//              for an id outside its table;
//   q_row[q]   output row b*T + t of the bag that holds id q;
// Steps (all on the caller's stream):
//   0. count    cnt[k] = number of valid pairs with counting key k = x & kmask
//               (cnt zeroed by the caller; k = x unless R exceeds the number
//               of counters, see SortedBuffers);
//   1. scan     start[k] = sum of cnt[y] for y < k (three kernels);
//               statistics: valid pairs and distinct keys;
//   2. scatter  each pair takes a slot in [start[k], start[k+1]) of sorted_e,
//               which holds (x, r = row*J + j): the bucket and the
//               upstream-gradient chunk to add (with signed hashing, bit 31 of
//               pair_x and of r carries the pair's sign, see pss_device.cuh);
//   3. reduce   the sorted entries are cut into tasks of kPiece consecutive
//               entries; one group of lanes per task owns 16-byte columns of
//               the block, adds the chunks of each run of equal x with
//               compensated (Kahan) fp32 sums, and adds every run's sum once
//               into the fp64 gradient accumulator g[G*x + z] -- one reduction
//               per run and element instead of one per contribution, and no
//               queue of reductions on a hot address.  With `mixed` (counters
//               shared by residue) runs of different buckets may alternate,
//               and a block of entries is summed as one run only when every
//               entry of it belongs to the current run.
// With counters shared by residue and the touched update, k_mark_pairs lists
// the touched blocks from pair_x (the scan cannot: a non-empty counter no
// longer names one bucket).
// The optimizer pass over g follows (pss_kernels.cu).
#include <climits>

#include "pss_device.cuh"
#include "pss_internal.h"

namespace pss {
namespace {

constexpr uint32_t kBad = 0xffffffffu;
constexpr int kScanThreads = 1024;
constexpr int kScanPerThread = 2;
constexpr int kScanChunk = kScanThreads * kScanPerThread;
constexpr int kRU = 4;            // entries in flight per group (summed as a tree when they
                                  // all continue the current run)
static_assert(kRU == 4, "the reduce sums kRU = 4 entries as a tree");

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
    pdl_prologue();
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
    pdl_prologue();
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
    pdl_prologue();
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

// Counting and slot assignment work on SEGMENTS of kSeg consecutive pairs,
// one per CTA at a time.  The CTA first merges its segment in a shared-memory
// hash table (bucket -> number of pairs; each pair's rank among the segment's
// pairs of its bucket), then touches the global counter of every DISTINCT
// bucket of the segment once.  Under a skewed (Zipf) id distribution a hot
// bucket therefore sees one global atomic per segment rather than one per
// pair, so no long queue of atomics forms on one address.
constexpr int kSegThreads = 256;
constexpr int kSegPer = 8;                        // pairs per thread
constexpr int kSeg = kSegThreads * kSegPer;       // pairs per segment
constexpr int kSegLog2Slots = 12;
constexpr int kSegSlots = 1 << kSegLog2Slots;     // hash slots (load factor <= 1/2)
static_assert(kSegSlots >= 2 * kSeg, "the segment table needs a free slot for every key");
static_assert(kSeg <= 65536 && kSegSlots <= 65536, "slot and rank are packed in 16 bits each");
constexpr int kSegFlushU = 4;                     // global atomics in flight per thread
constexpr uint32_t kEmpty = 0xffffffffu;          // == kBad, which is never inserted

// Insert bucket x (not kBad) into the segment table; returns the slot in the
// low 16 bits and the pair's rank among the segment's pairs of bucket x in
// the high 16 bits.  Linear probing always ends: the table has more slots
// than a segment has pairs.
__device__ __forceinline__ uint32_t seg_insert(uint32_t* s_key, uint32_t* s_val, uint32_t x) {
    uint32_t h = (x * 0x9e3779b1u) >> (32 - kSegLog2Slots);
    for (int probe = 0; probe < kSegSlots; ++probe) {
        const uint32_t prev = atomicCAS(s_key + h, kEmpty, x);
        if (prev == kEmpty || prev == x) break;
        h = (h + 1u) & (uint32_t)(kSegSlots - 1);
    }
    return h | (atomicAdd(s_val + h, 1u) << 16);
}

__device__ __forceinline__ void seg_table_init(uint32_t* s_key, uint32_t* s_val) {
    for (int i = threadIdx.x; i < kSegSlots; i += kSegThreads) {
        s_key[i] = kEmpty;
        s_val[i] = 0u;
    }
}

// cnt[k] += number of valid pairs with counting key k = (x without its sign) & kmask.
__global__ void __launch_bounds__(kSegThreads)
k_sort_count(const uint32_t* __restrict__ pair_x, int64_t npairs, uint32_t smask, uint32_t kmask,
             uint32_t* __restrict__ cnt) {
    pdl_prologue();
    __shared__ uint32_t s_key[kSegSlots];
    __shared__ uint32_t s_val[kSegSlots];
    seg_table_init(s_key, s_val);
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    for (int64_t seg = blockIdx.x; seg < nseg; seg += gridDim.x) {
        const int64_t p0 = seg * kSeg;
        uint32_t x[kSegPer], hr[kSegPer];
#pragma unroll
        for (int i = 0; i < kSegPer; ++i) {
            const int64_t p = p0 + i * kSegThreads + threadIdx.x;
            x[i] = (p < npairs) ? __ldg(pair_x + p) : kBad;
        }
        __syncthreads();   // the previous segment's table is clear
#pragma unroll
        for (int i = 0; i < kSegPer; ++i)
            hr[i] = (x[i] != kBad) ? seg_insert(s_key, s_val, x[i] & ~smask & kmask) : 0u;
        __syncthreads();
#pragma unroll
        for (int k = 0; k < kSegSlots / kSegThreads; ++k) {
            const int sl = k * kSegThreads + threadIdx.x;
            const uint32_t key = s_key[sl];
            if (key != kEmpty) atomicAdd(cnt + key, s_val[sl]);
        }
        __syncthreads();
        // each thread clears the slots of its own pairs
#pragma unroll
        for (int i = 0; i < kSegPer; ++i)
            if (x[i] != kBad) {
                s_key[hr[i] & 0xffffu] = kEmpty;
                s_val[hr[i] & 0xffffu] = 0u;
            }
    }
}

// Slot of every valid pair: cnt counts back down to zero, each segment taking
// one contiguous range of its counting key for every bucket it holds (one
// atomic per distinct bucket); within the range a pair's place is its rank in
// the segment table, which is keyed by the bucket, so a segment's pairs of one
// bucket stay together even when several buckets share a key.
// sorted_e[slot] = x << 32 | row*J + j.
template <bool SG>
__global__ void __launch_bounds__(kSegThreads)
k_sort_scatter(const uint32_t* __restrict__ pair_x, int64_t npairs, const uint32_t* __restrict__ q_row,
               int J, int log2J, uint32_t kmask, const uint32_t* __restrict__ start,
               uint32_t* __restrict__ cnt, unsigned long long* __restrict__ sorted_e) {
    pdl_prologue();
    __shared__ uint32_t s_key[kSegSlots];
    __shared__ uint32_t s_val[kSegSlots];
    seg_table_init(s_key, s_val);
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    for (int64_t seg = blockIdx.x; seg < nseg; seg += gridDim.x) {
        const int64_t p0 = seg * kSeg;
        uint32_t x[kSegPer], hr[kSegPer], e[kSegPer], st0[kSegPer];
#pragma unroll
        for (int i = 0; i < kSegPer; ++i) {
            const int64_t p = p0 + i * kSegThreads + threadIdx.x;
            x[i] = (p < npairs) ? __ldg(pair_x + p) : kBad;
        }
        // loads that do not depend on the table go first, so they overlap it
#pragma unroll
        for (int i = 0; i < kSegPer; ++i) {
            const uint32_t pp = (uint32_t)(p0 + i * kSegThreads + threadIdx.x);  // npairs < 2^32 here
            const uint32_t q = (log2J >= 0) ? (pp >> log2J) : pp / (uint32_t)J;
            e[i] = pp - q * (uint32_t)J;
            st0[i] = 0u;
            if (x[i] != kBad) {
                e[i] += __ldg(q_row + q) * (uint32_t)J;
                if (SG) {
                    // signed hashing: the sign moves to bit 31 of the entry's low word
                    e[i] |= x[i] & 0x80000000u;
                    x[i] &= 0x7fffffffu;
                }
                st0[i] = __ldg(start + (x[i] & kmask));
            }
        }
        __syncthreads();   // the previous segment's table is clear
#pragma unroll
        for (int i = 0; i < kSegPer; ++i)
            hr[i] = (x[i] != kBad) ? seg_insert(s_key, s_val, x[i]) : 0u;
        __syncthreads();
        // one countdown per distinct bucket, kSegFlushU in flight per thread;
        // the slot's value becomes the segment's first place in the bucket
#pragma unroll
        for (int k0 = 0; k0 < kSegSlots / kSegThreads; k0 += kSegFlushU) {
            uint32_t key[kSegFlushU], c[kSegFlushU], old[kSegFlushU];
#pragma unroll
            for (int u = 0; u < kSegFlushU; ++u) {
                const int sl = (k0 + u) * kSegThreads + threadIdx.x;
                key[u] = s_key[sl];
                c[u] = s_val[sl];
            }
#pragma unroll
            for (int u = 0; u < kSegFlushU; ++u)
                old[u] = (key[u] != kEmpty) ? atomicSub(cnt + (key[u] & kmask), c[u]) : 0u;
#pragma unroll
            for (int u = 0; u < kSegFlushU; ++u)
                if (key[u] != kEmpty) s_val[(k0 + u) * kSegThreads + threadIdx.x] = old[u] - c[u];
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kSegPer; ++i) {
            if (x[i] == kBad) continue;
            const uint32_t slot = st0[i] + s_val[hr[i] & 0xffffu] + (hr[i] >> 16);
            sorted_e[slot] = ((unsigned long long)x[i] << 32) | e[i];
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kSegPer; ++i)
            if (x[i] != kBad) {
                s_key[hr[i] & 0xffffu] = kEmpty;
                s_val[hr[i] & 0xffffu] = 0u;
            }
    }
}

// Touched bitmap and list of the buckets of all valid pairs.  A CTA takes
// chunks of kMarkChunk pairs; a bucket already marked costs one load, a new
// one an atomicOr, and the CTA gathers its new buckets in shared memory and
// reserves their list places with one atomic per chunk.
constexpr int kMarkPer = 16;                          // pairs per thread and chunk
constexpr int kMarkChunk = kThreads * kMarkPer;

__global__ void __launch_bounds__(kThreads)
k_mark_pairs(const uint32_t* __restrict__ pair_x, int64_t npairs, uint32_t smask, Touched tc) {
    pdl_prologue();
    __shared__ uint32_t s_new[kMarkChunk];
    __shared__ uint32_t s_n;
    __shared__ unsigned long long s_base;
    const int64_t nchunks = (npairs + kMarkChunk - 1) / kMarkChunk;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
        if (threadIdx.x == 0) s_n = 0u;
        __syncthreads();
        uint32_t x[kMarkPer], word[kMarkPer];
#pragma unroll
        for (int i = 0; i < kMarkPer; ++i) {
            const int64_t p = c * kMarkChunk + i * kThreads + threadIdx.x;
            x[i] = (p < npairs) ? __ldg(pair_x + p) : kBad;
        }
#pragma unroll
        for (int i = 0; i < kMarkPer; ++i) {
            if (x[i] != kBad) x[i] &= ~smask;
            word[i] = (x[i] != kBad) ? __ldcg(tc.bitmap + (x[i] >> 5)) : ~0u;
        }
#pragma unroll
        for (int i = 0; i < kMarkPer; ++i) {
            const uint32_t bit = 1u << (x[i] & 31u);
            if (!(word[i] & bit) && !(atomicOr(tc.bitmap + (x[i] >> 5), bit) & bit))
                s_new[atomicAdd(&s_n, 1u)] = x[i];
        }
        __syncthreads();
        const uint32_t n = s_n;
        if (threadIdx.x == 0) s_base = n ? atomicAdd(tc.count, (unsigned long long)n) : 0ull;
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < n; k += kThreads) {
            const unsigned long long slot = s_base + k;
            if ((int64_t)slot < tc.cap) tc.list[slot] = (int64_t)s_new[k];
        }
        __syncthreads();   // s_new and s_n are reused by the next chunk
    }
}

// Reduce: one group of gs lanes per task of kPiece sorted entries; lane lg
// owns columns lg + k*gs of VW elements of the L-element block.  Each run of
// equal x is summed with compensation (Kahan) and added once into the fp64
// accumulator through a shared-memory transpose (so that every fp64
// reduction instruction covers consecutive elements).
constexpr int64_t kPiece = 64;    // sorted entries per reduce task

template <int VW, int KC, bool JPOW2, bool ZDIV>
__global__ void __launch_bounds__(kThreads, (KC == 1) ? 4 : 1)
k_range_reduce(const unsigned long long* __restrict__ sorted_e,
               const unsigned long long* __restrict__ stats, int64_t npairs,
               const float* __restrict__ gout, int d, int Z, int J, int log2J, int L, int64_t G,
               uint32_t smask, bool mixed, double* __restrict__ g, int log2gs) {
    pdl_prologue();
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
    int colk[KC];
#pragma unroll
    for (int k = 0; k < KC; ++k) colk[k] = (lg + k * gs) * VW;
    float s[KC][VW], c[KC][VW];

    auto flush = [&](uint32_t x) {
#pragma unroll
        for (int k = 0; k < KC; ++k) {
#pragma unroll
            for (int i = 0; i < VW; ++i) {
                if (colk[k] + i < L) stage[colk[k] + i] = s[k][i];
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
                const uint32_t r = (uint32_t)ent[u] & ~smask;
                const uint32_t sb = (uint32_t)ent[u] & smask;
                if (xs[u] != kBad) {
                    if (ZDIV) {
                        // Z divides d: chunk r starts at r*Z and is Z long
                        const float* src = gout + (uint64_t)r * (uint64_t)Z;
#pragma unroll
                        for (int k = 0; k < KC; ++k) {
                            if (colk[k] < L) v[u][k] = sign_by(V::ldcs(src + colk[k]), sb);
                            else
#pragma unroll
                                for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                        }
                    } else {
                        const uint32_t row = JPOW2 ? (r >> log2J) : r / (uint32_t)J;
                        const int j = (int)(r - row * (uint32_t)J);
                        const int Lj = (d - j * Z) < Z ? (d - j * Z) : Z;
                        const float* src = gout + (int64_t)row * d + j * Z;
#pragma unroll
                        for (int k = 0; k < KC; ++k) {
                            if (colk[k] < Lj) v[u][k] = sign_by(V::ldcs(src + colk[k]), sb);
                            else
#pragma unroll
                                for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                        }
                    }
                } else {
#pragma unroll
                    for (int k = 0; k < KC; ++k)
#pragma unroll
                        for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                }
            }
            // the whole block continues the current run when its last entry
            // does (entries in bucket order), or, when runs of buckets that
            // share a counting key may alternate, when every entry does
            if (xs[kRU - 1] == cur &&
                (!mixed || (xs[0] == cur && xs[1] == cur && xs[2] == cur))) {
                // a tree sum, then one compensated add
#pragma unroll
                for (int k = 0; k < KC; ++k)
#pragma unroll
                    for (int i = 0; i < VW; ++i) {
                        const float a01 = V::get(v[0][k], i) + V::get(v[1][k], i);
                        const float a23 = V::get(v[2][k], i) + V::get(v[3][k], i);
                        kahan_add(s[k][i], c[k][i], a01 + a23);
                    }
            } else {
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
                        for (int i = 0; i < VW; ++i)
                            kahan_add(s[k][i], c[k][i], V::get(v[u][k], i));
                }
            }
        }
        flush(cur);
    }
}

// Reduce for blocks of at least 32 elements: one WARP per task of kPiece
// sorted entries, lane z owning elements z, z+32, ... of the block, so every
// branch is warp-uniform and a run's sum goes straight from the lanes to the
// fp64 accumulator (32 consecutive doubles per instruction).  The task's
// entries are staged in shared memory with one coalesced load; kWU chunk
// loads per lane are in flight; a block of kWU entries that continues the
// current run is summed as a tree and added with compensation once.
constexpr int kWU = 8;
static_assert(kWU == 8, "the warp reduce sums kWU = 8 entries as a tree");

template <int KE, bool ZDIV, bool JPOW2>
__global__ void __launch_bounds__(kThreads)
k_warp_range_reduce(const unsigned long long* __restrict__ sorted_e,
                    const unsigned long long* __restrict__ stats, int64_t npairs,
                    const float* __restrict__ gout, int d, int Z, int J, int log2J, int L,
                    int64_t G, uint32_t smask, bool mixed, double* __restrict__ g) {
    pdl_prologue();
    __shared__ unsigned long long s_ent[kWarps][kPiece];
    const int64_t total = (int64_t)(stats[0] < (unsigned long long)npairs ? stats[0] : npairs);
    const int64_t ntasks = (total + kPiece - 1) / kPiece;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    unsigned long long* ent = s_ent[warp];
    const int64_t wstride = (int64_t)gridDim.x * kWarps;
    constexpr unsigned long long kNone = (unsigned long long)kBad << 32;
    float s[KE], c[KE];
    auto flush = [&](uint32_t x) {
        double* base = g + (int64_t)x * G;
#pragma unroll
        for (int k = 0; k < KE; ++k) {
            const int z = lane + 32 * k;
            if (z < L && s[k] != 0.f) red_add_f64(base + z, widen(s[k]));
            s[k] = c[k] = 0.f;
        }
    };
    for (int64_t t = (int64_t)blockIdx.x * kWarps + warp; t < ntasks; t += wstride) {
        const int64_t e0 = t * kPiece;
        const int n = (int)((e0 + kPiece < total) ? kPiece : total - e0);
#pragma unroll
        for (int h = 0; h < (int)kPiece; h += 32)
            ent[h + lane] = (h + lane < n) ? __ldg(sorted_e + e0 + h + lane) : kNone;
        __syncwarp();
#pragma unroll
        for (int k = 0; k < KE; ++k) s[k] = c[k] = 0.f;
        uint32_t cur = (uint32_t)(ent[0] >> 32);
        for (int b = 0; b < n; b += kWU) {
            uint32_t xs[kWU];
            float v[kWU][KE];
#pragma unroll
            for (int u = 0; u < kWU; ++u) {
                const unsigned long long en = ent[b + u < (int)kPiece ? b + u : (int)kPiece - 1];
                xs[u] = (b + u < n) ? (uint32_t)(en >> 32) : kBad;
                const uint32_t r = (uint32_t)en & ~smask;
                const uint32_t sb = (uint32_t)en & smask;
                const float* src;
                int Lj;
                if (ZDIV) {
                    src = gout + (uint64_t)r * (uint64_t)Z;
                    Lj = L;
                } else {
                    const uint32_t row = JPOW2 ? (r >> log2J) : r / (uint32_t)J;
                    const int j = (int)(r - row * (uint32_t)J);
                    Lj = (d - j * Z) < Z ? (d - j * Z) : Z;
                    src = gout + (int64_t)row * d + j * Z;
                }
#pragma unroll
                for (int k = 0; k < KE; ++k) {
                    const int z = lane + 32 * k;
                    v[u][k] = (xs[u] != kBad && z < Lj) ? sign_by(__ldcs(src + z), sb) : 0.f;
                }
            }
            bool cont = xs[kWU - 1] == cur;
            if (mixed) {
#pragma unroll
                for (int u = 0; u < kWU - 1; ++u) cont = cont && xs[u] == cur;
            }
            if (cont) {
#pragma unroll
                for (int k = 0; k < KE; ++k) {
                    const float a = (v[0][k] + v[1][k]) + (v[2][k] + v[3][k]);
                    const float bsum = (v[4][k] + v[5][k]) + (v[6][k] + v[7][k]);
                    kahan_add(s[k], c[k], a + bsum);
                }
            } else {
#pragma unroll
                for (int u = 0; u < kWU; ++u) {
                    if (xs[u] == kBad) break;
                    if (xs[u] != cur) {
                        flush(cur);
                        cur = xs[u];
                    }
#pragma unroll
                    for (int k = 0; k < KE; ++k) kahan_add(s[k], c[k], v[u][k]);
                }
            }
        }
        flush(cur);
        __syncwarp();
    }
}

// Reduce for 32-element chunks that tile the rows (Z = 32 dividing d): the
// upstream-gradient chunks of a warp's task are staged asynchronously into
// shared memory (cp.async, 16 bytes per lane), kAD - 1 stages of kAS chunks in
// flight per warp, so the data in flight is bounded by shared memory rather
// than registers.  Lane z then sums element z of each chunk (compensated; a
// stage that continues the current run is summed as a tree first) and adds
// every run's sum once into the fp64 accumulator.
constexpr int kAS = 8;          // chunks per stage
constexpr int kAD = 4;          // ring slots (kAD - 1 stages in flight)
// sorted entries per task.  Measured: 256 gave the multi-hot reduce 0.254
// against 0.268 ms and left the Criteo-TB one unchanged, but its 48 KB of
// shared memory allow one CTA less per SM and a batch of 16384 leaves ~1.4
// tasks per warp: that reduce took 77 against 57 us.
constexpr int kAPiece = 128;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" :: "r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" :: "n"(N) : "memory");
}

__global__ void __launch_bounds__(kThreads)
k_async_reduce(const unsigned long long* __restrict__ sorted_e,
               const unsigned long long* __restrict__ stats, int64_t npairs,
               const float* __restrict__ gout, int64_t G, uint32_t smask, bool mixed,
               double* __restrict__ g) {
    pdl_prologue();
    __shared__ __align__(16) float s_ring[kWarps][kAD][kAS][32];
    __shared__ unsigned long long s_ent[kWarps][kAPiece];
    const int64_t total = (int64_t)(stats[0] < (unsigned long long)npairs ? stats[0] : npairs);
    const int64_t ntasks = (total + kAPiece - 1) / kAPiece;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    unsigned long long* ent = s_ent[warp];
    const int64_t wstride = (int64_t)gridDim.x * kWarps;
    constexpr unsigned long long kNone = (unsigned long long)kBad << 32;
    float sum = 0.f, comp = 0.f;
    auto flush = [&](uint32_t x) {
        if (sum != 0.f) red_add_f64(g + (int64_t)x * G + lane, widen(sum));
        sum = comp = 0.f;
    };
    for (int64_t t = (int64_t)blockIdx.x * kWarps + warp; t < ntasks; t += wstride) {
        const int64_t e0 = t * kAPiece;
        const int n = (int)((e0 + kAPiece < total) ? kAPiece : total - e0);
#pragma unroll
        for (int h = 0; h < kAPiece; h += 32)
            ent[h + lane] = (h + lane < n) ? __ldg(sorted_e + e0 + h + lane) : kNone;
        __syncwarp();
        const int nst = (n + kAS - 1) / kAS;
        // copy stage st (kAS chunks of 128 bytes = 64 pieces of 16 bytes)
        auto issue = [&](int st) {
            if (st < nst) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int pc = lane + 32 * h;
                    const int i = pc >> 3;
                    const int part = pc & 7;
                    const int e = st * kAS + i;
                    if (e < n) {
                        const uint32_t r =
                            reinterpret_cast<const uint32_t*>(ent)[2 * e] & ~smask;  // low word
                        cp_async16(&s_ring[warp][st % kAD][i][part * 4],
                                   gout + (uint64_t)r * 32u + (uint32_t)(part * 4));
                    }
                }
            }
            cp_async_commit();
        };
#pragma unroll
        for (int st = 0; st < kAD - 1; ++st) issue(st);
        sum = comp = 0.f;
        uint32_t cur = (uint32_t)(ent[0] >> 32);
        for (int st = 0; st < nst; ++st) {
            issue(st + kAD - 1);
            cp_async_wait<kAD - 1>();
            __syncwarp();
            const float* buf = &s_ring[warp][st % kAD][0][0];
            const uint32_t* ex = reinterpret_cast<const uint32_t*>(ent + st * kAS) + 1;  // high words: x
            // the entries are sorted and padded with kBad: when the stage's last
            // bucket continues the run, the stage is full and all of it does
            // all loads first, in one round trip (the flush's reduction is a
            // memory barrier for the compiler, so later loads would not overlap);
            // chunks past the task's end are never read as values
            const uint32_t xlast = ex[2 * (kAS - 1)];
            float v[kAS];
#pragma unroll
            for (int i = 0; i < kAS; ++i) v[i] = buf[i * 32 + lane];
            if (smask) {
                // signed hashing: each entry's sign is bit 31 of its low word
#pragma unroll
                for (int i = 0; i < kAS; ++i) v[i] = sign_by(v[i], ex[2 * i - 1] & smask);
            }
            // with alternating runs (buckets sharing a counting key) every
            // entry of the stage is compared, one per lane
            const bool cont =
                xlast == cur &&
                (!mixed || __all_sync(0xffffffffu, ex[2 * (lane & (kAS - 1))] == cur));
            if (cont) {
                const float a = (v[0] + v[1]) + (v[2] + v[3]);
                const float b = (v[4] + v[5]) + (v[6] + v[7]);
                kahan_add(sum, comp, a + b);
            } else {
                uint32_t xs[kAS];
#pragma unroll
                for (int i = 0; i < kAS; ++i) xs[i] = ex[2 * i];
#pragma unroll
                for (int i = 0; i < kAS; ++i) {
                    if (xs[i] == kBad) break;
                    if (xs[i] != cur) {
                        flush(cur);
                        cur = xs[i];
                    }
                    kahan_add(sum, comp, v[i]);
                }
            }
            __syncwarp();
        }
        flush(cur);
        cp_async_wait<0>();
        __syncwarp();
    }
}

template <int KE, bool ZDIV, bool JPOW2>
cudaError_t warp_reduce_launch(const SortedBuffers& sb, int64_t npairs, const float* gout,
                               const DevParams& p, double* g, int log2J, int sm_count,
                               cudaStream_t st) {
    const int64_t ntasks = (npairs + kPiece - 1) / kPiece;   // upper bound
    const int grid = grid_for(k_warp_range_reduce<KE, ZDIV, JPOW2>, sm_count,
                              (ntasks + kWarps - 1) / kWarps);
    return launch_k(k_warp_range_reduce<KE, ZDIV, JPOW2>, dim3(grid), dim3(kThreads), 0, st,
                    sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, log2J, p.L, p.G, p.smask,
                    sb.kmask != 0xffffffffu, g);
}

template <int KE>
cudaError_t warp_reduce_inst(const SortedBuffers& sb, int64_t npairs, const float* gout,
                             const DevParams& p, double* g, int sm_count, cudaStream_t st) {
    const int log2J = (p.J & (p.J - 1)) == 0 ? ceil_log2(p.J) : -1;
    if (p.d % p.Z == 0)
        return warp_reduce_launch<KE, true, true>(sb, npairs, gout, p, g, 0, sm_count, st);
    if (log2J >= 0)
        return warp_reduce_launch<KE, false, true>(sb, npairs, gout, p, g, log2J, sm_count, st);
    return warp_reduce_launch<KE, false, false>(sb, npairs, gout, p, g, 0, sm_count, st);
}

template <int VW, int KC, bool JPOW2, bool ZDIV>
cudaError_t reduce_launch(const SortedBuffers& sb, int64_t npairs, const float* gout,
                          const DevParams& p, double* g, int log2J, int log2gs, int sm_count,
                          cudaStream_t st) {
    const int gpc = kWarps * (32 >> log2gs);
    const size_t smem = sizeof(float) * (size_t)gpc * (size_t)p.L;
    const int64_t ntasks = (npairs + kPiece - 1) / kPiece;   // upper bound
    const int64_t work_blocks = (ntasks + gpc - 1) / gpc;
    const int grid = grid_for(k_range_reduce<VW, KC, JPOW2, ZDIV>, sm_count, work_blocks, smem);
    return launch_k(k_range_reduce<VW, KC, JPOW2, ZDIV>, dim3(grid), dim3(kThreads), smem, st,
                    sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, log2J, p.L, p.G, p.smask,
                    sb.kmask != 0xffffffffu, g, log2gs);
}

template <int VW, int KC>
cudaError_t reduce_inst(const SortedBuffers& sb, int64_t npairs, const float* gout,
                        const DevParams& p, double* g, int log2gs, int sm_count,
                        cudaStream_t st) {
    const int log2J = (p.J & (p.J - 1)) == 0 ? ceil_log2(p.J) : -1;
    if (p.d % p.Z == 0)
        return reduce_launch<VW, KC, true, true>(sb, npairs, gout, p, g, 0, log2gs, sm_count, st);
    if (log2J >= 0)
        return reduce_launch<VW, KC, true, false>(sb, npairs, gout, p, g, log2J, log2gs, sm_count,
                                                  st);
    return reduce_launch<VW, KC, false, false>(sb, npairs, gout, p, g, 0, log2gs, sm_count, st);
}

}  // namespace

int64_t sorted_scan_blocks(int64_t R) { return (R + kScanChunk - 1) / kScanChunk; }



cudaError_t launch_sorted_scan(const SortedBuffers& sb, int64_t R, const Touched* touched,
                               cudaStream_t st) {
    const int64_t nblk = sorted_scan_blocks(R);
    const Touched tc = touched ? *touched : Touched{};
    cudaError_t e = launch_k(k_scan_reduce, dim3((unsigned)nblk), dim3(kScanThreads), 0, st,
                             sb.cnt, R, sb.bsum, sb.bnz);
    if (e != cudaSuccess) return e;
    e = launch_k(k_scan_top, dim3(1), dim3(kScanThreads), 0, st, sb.bsum, sb.bnz, nblk, sb.stats,
                 tc.count);
    if (e != cudaSuccess) return e;
    return launch_k(k_scan_apply, dim3((unsigned)nblk), dim3(kScanThreads), 0, st, sb.cnt, R,
                    sb.bsum, sb.bnz, sb.start, tc);
}

cudaError_t launch_sorted_scatter(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                                  int sm_count, cudaStream_t st) {
    const int log2J = (J & (J - 1)) == 0 ? ceil_log2(J) : -1;
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    if (smask) {
        const int grid = grid_for(k_sort_scatter<true>, sm_count, nseg);
        return launch_k(k_sort_scatter<true>, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x,
                        npairs, sb.q_row, J, log2J, sb.kmask, sb.start, sb.cnt, sb.sorted_e);
    }
    const int grid = grid_for(k_sort_scatter<false>, sm_count, nseg);
    return launch_k(k_sort_scatter<false>, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x, npairs,
                    sb.q_row, J, log2J, sb.kmask, sb.start, sb.cnt, sb.sorted_e);
}

cudaError_t launch_sorted_count(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                                int sm_count, cudaStream_t st) {
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    const int grid = grid_for(k_sort_count, sm_count, nseg);
    return launch_k(k_sort_count, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x, npairs, smask,
                    sb.kmask, sb.cnt);
}

cudaError_t launch_mark_pairs(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                              const Touched& touched, int sm_count, cudaStream_t st) {
    const int64_t chunks = (npairs + kMarkChunk - 1) / kMarkChunk;
    const int grid = grid_for(k_mark_pairs, sm_count, chunks);
    return launch_k(k_mark_pairs, dim3(grid), dim3(kThreads), 0, st, sb.pair_x, npairs, smask,
                    touched);
}

cudaError_t launch_sorted_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, double* g, int sm_count, cudaStream_t st) {
    // 32-element chunks tiling the rows: asynchronous shared-memory staging
    if (p.Z == 32 && p.d % 32 == 0 && (((uintptr_t)gout & 15u) == 0)) {
        const int64_t ntasks = (npairs + kAPiece - 1) / kAPiece;   // upper bound
        const int grid = grid_for(k_async_reduce, sm_count, (ntasks + kWarps - 1) / kWarps);
        return launch_k(k_async_reduce, dim3(grid), dim3(kThreads), 0, st, sb.sorted_e, sb.stats,
                        npairs, gout, p.G, p.smask, sb.kmask != 0xffffffffu, g);
    }
    // blocks of 32+ elements: one warp per task, one element per lane
    if (p.L >= 32) {
        if (p.L <= 32) return warp_reduce_inst<1>(sb, npairs, gout, p, g, sm_count, st);
        if (p.L <= 64) return warp_reduce_inst<2>(sb, npairs, gout, p, g, sm_count, st);
        if (p.L <= 128) return warp_reduce_inst<4>(sb, npairs, gout, p, g, sm_count, st);
    }
    const bool vec = (p.Z % 4 == 0) && (p.d % 4 == 0) && (((uintptr_t)gout & 15u) == 0);
    const int vw = vec ? 4 : 1;
    const int V = (p.L + vw - 1) / vw;
    const int log2gs = V <= 32 ? ceil_log2(V) : 5;
    const int kc = V <= 32 ? 1 : (1 << ceil_log2((V + 31) / 32));
#define PSS_RD(VW, KC) return reduce_inst<VW, KC>(sb, npairs, gout, p, g, log2gs, sm_count, st)
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
