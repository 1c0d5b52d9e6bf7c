// Sorted backward path (the sparse branch of Algorithm 1: find the distinct
// locations, sum the contributions of each, then apply them).
//
// Input, written by the forward pass of the same batch:
//   pair_x[p]  bucket x of pair p = q*J + j (block start G*x), or 0xffffffff
//              for an id outside its table;
//   q_row[q]   output row b*T + t of the bag that holds id q;
// Steps (all on the caller's stream):
//   1. sort     a stable radix sort of the entries e = x << 32 | r by x, where
//               r = row*J + j names the upstream-gradient chunk to add (with
//               signed hashing, bit 31 of pair_x and of r carries the pair's
//               sign, see pss_device.cuh); bad ids are dropped.  Entries of one
//               bucket come out in pair order, so every later step sees the
//               same sequence on every run;
//   2. reduce   the sorted entries are cut into tasks of consecutive entries;
//               the lanes of a task own columns of the block, add the chunks of
//               each run of equal x with compensated (Kahan) fp32 sums, and add
//               every run's sum once into the fp64 gradient accumulator
//               g[G*x + z] -- one reduction per run and element instead of one
//               per contribution, and no queue of reductions on a hot address.
//               The distinct buckets (stats[1]) come from the counting sort's
//               scan, or, after a radix sort, from the reduce.
// With the touched update, k_mark_pairs lists the touched blocks from pair_x.
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

// ---------------------------------------------------------------------------
// Counting sort by bucket (the default when R <= kCountSortMaxR): a count of
// every bucket, a scan of the counts (two kernels), and a slot scatter.
// Every bucket has its own counter, so the entries come out grouped by bucket;
// their order inside a bucket depends on the GPU's scheduling.
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

// start[x] = exclusive prefix of cnt; start[R] = total; cnt returns to zero
// for the next sort's count.  Each block first adds up the chunk sums of the
// blocks before it (a few hundred values).  The last block writes stats[0] =
// valid pairs and stats[1] = distinct buckets (non-empty counters).
// With a touched list, the non-empty buckets are listed in order and their
// bits set, and the last block writes the list's length.
__global__ void __launch_bounds__(kScanThreads)
k_scan_apply(uint32_t* __restrict__ cnt, int64_t R, const uint32_t* __restrict__ bsum,
             const uint32_t* __restrict__ bnz, uint32_t* __restrict__ start, Touched tc,
             unsigned long long* __restrict__ stats) {
    pdl_prologue();
    __shared__ uint32_t s_warp[33];
    const int64_t base = (int64_t)blockIdx.x * kScanChunk;
    uint32_t pv = 0u, pz = 0u;
    for (int64_t b = threadIdx.x; b < (int64_t)blockIdx.x; b += kScanThreads) {
        pv += bsum[b];
        pz += bnz[b];
    }
    uint32_t pre_v, pre_z;
    block_exclusive_scan(pv, s_warp, &pre_v);
    block_exclusive_scan(pz, s_warp, &pre_z);
    uint32_t c[kScanPerThread];
    uint32_t sum = 0, nz = 0;
#pragma unroll
    for (int i = 0; i < kScanPerThread; ++i) {
        const int64_t e = base + (int64_t)threadIdx.x * kScanPerThread + i;
        c[i] = (e < R) ? cnt[e] : 0u;
        if (e < R && c[i]) cnt[e] = 0u;
        sum += c[i];
        nz += (c[i] != 0u);
    }
    uint32_t tot_v, tot_z;
    uint32_t run = pre_v + block_exclusive_scan(sum, s_warp, &tot_v);
    uint32_t zrun = pre_z + block_exclusive_scan(nz, s_warp, &tot_z);
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
        stats[0] = pre_v + tot_v;
        stats[1] = pre_z + tot_z;   // distinct buckets: the non-empty counters
        if (tc.count) *tc.count = pre_z + tot_z;
    }
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
// Segments of 1024 pairs in 2048 slots: measured on GB300 at the Criteo-TB
// shape, count + scan + scatter took 0.124 ms against 0.145 with 2048 pairs
// in 4096 slots, 0.150 with 1024 pairs in 4096 slots and 0.125 with 512 in
// 1024 (multi-hot shape: 0.227, 0.258, -, 0.247 ms); the scans of the table
// that the count and the atomics take cost in proportion to its slots.
constexpr int kSegThreads = 256;
constexpr int kSegPer = 4;                        // pairs per thread
constexpr int kSeg = kSegThreads * kSegPer;       // pairs per segment
constexpr int kSegLog2Slots = 11;
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

// cnt[x] += number of valid pairs with bucket x (without its sign).
__global__ void __launch_bounds__(kSegThreads)
k_sort_count(const uint32_t* __restrict__ pair_x, int64_t npairs, uint32_t smask,
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
            hr[i] = (x[i] != kBad) ? seg_insert(s_key, s_val, x[i] & ~smask) : 0u;
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

// Slot of every valid pair: start[x] serves as bucket x's next free place,
// each segment taking one contiguous range of the bucket for every bucket it
// holds (one atomic per distinct bucket, which returns the range's first
// place); within the range a pair's place is its rank in the segment table.
// Which segment takes which range, and the ranks, follow the order in which
// the GPU runs the atomics.  start[x] ends at the bucket's end.
// sorted_e[slot] = x << 32 | row*J + j.
template <bool SG>
__global__ void __launch_bounds__(kSegThreads)
k_sort_scatter(const uint32_t* __restrict__ pair_x, int64_t npairs, const uint32_t* __restrict__ q_row,
               int J, int log2J, uint32_t* __restrict__ start,
               unsigned long long* __restrict__ sorted_e) {
    pdl_prologue();
    __shared__ uint32_t s_key[kSegSlots];
    __shared__ uint32_t s_val[kSegSlots];
    seg_table_init(s_key, s_val);
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    for (int64_t seg = blockIdx.x; seg < nseg; seg += gridDim.x) {
        const int64_t p0 = seg * kSeg;
        uint32_t x[kSegPer], hr[kSegPer], e[kSegPer];
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
            if (x[i] != kBad) {
                e[i] += __ldg(q_row + q) * (uint32_t)J;
                if (SG) {
                    // signed hashing: the sign moves to bit 31 of the entry's low word
                    e[i] |= x[i] & 0x80000000u;
                    x[i] &= 0x7fffffffu;
                }
            }
        }
        __syncthreads();   // the previous segment's table is clear
#pragma unroll
        for (int i = 0; i < kSegPer; ++i)
            hr[i] = (x[i] != kBad) ? seg_insert(s_key, s_val, x[i]) : 0u;
        __syncthreads();
        // one atomic per distinct bucket, kSegFlushU in flight per thread;
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
                old[u] = (key[u] != kEmpty) ? atomicAdd(start + key[u], c[u]) : 0u;
#pragma unroll
            for (int u = 0; u < kSegFlushU; ++u)
                if (key[u] != kEmpty) s_val[(k0 + u) * kSegThreads + threadIdx.x] = old[u];
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kSegPer; ++i) {
            if (x[i] == kBad) continue;
            const uint32_t slot = s_val[hr[i] & 0xffffu] + (hr[i] >> 16);
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

// ---------------------------------------------------------------------------
// Segment-local sort.  The pairs are cut into segments of kLS consecutive
// pairs, and each segment's valid entries are grouped by bucket inside the
// segment's own range of sorted_e, [s*kLS, s*kLS + segn[s]): no counter per
// bucket, no scan over all R buckets, no global atomics.  A bucket that occurs
// in several segments then has one run in each; the reduce adds every run's
// sum into the fp64 accumulator, so each element receives the same sum,
// grouped differently.  Consecutive pairs are consecutive ids of one table,
// so a segment merges the repeats of the table's hot ids (under Zipf ids the
// ones that would otherwise queue reductions on one address).
//
// Within a segment: every thread inserts its pairs into a shared-memory hash
// table (bucket -> count; each pair's rank among the segment's pairs of its
// bucket), the slot counts are scanned in a fixed slot order, and a pair goes
// to its slot's start plus its rank.  Which pair of a bucket comes first
// follows the order of the shared-memory atomics.
constexpr int kLSLog2 = 13;
constexpr int kLS = 1 << kLSLog2;                 // pairs per segment (8192)
constexpr int kLSThreads = 1024;
constexpr int kLSPer = kLS / kLSThreads;          // pairs per thread
constexpr int kLSLog2Slots = kLSLog2 + 1;         // load factor <= 1/2
constexpr int kLSSlots = 1 << kLSLog2Slots;
constexpr int kLSSlotsPer = kLSSlots / kLSThreads;
static_assert(kLS <= 65536 && kLSSlots <= 65536, "slot and rank are packed in 16 bits each");
static_assert(kLSThreads == kScanThreads, "the local sort scans with block_exclusive_scan");

__device__ __forceinline__ uint32_t local_insert(uint32_t* s_key, uint32_t* s_val, uint32_t x) {
    uint32_t h = (x * 0x9e3779b1u) >> (32 - kLSLog2Slots);
    for (int probe = 0; probe < kLSSlots; ++probe) {
        const uint32_t prev = atomicCAS(s_key + h, kEmpty, x);
        if (prev == kEmpty || prev == x) break;
        h = (h + 1u) & (uint32_t)(kLSSlots - 1);
    }
    return h | (atomicAdd(s_val + h, 1u) << 16);
}

// sorted_e[s*kLS + pos] = x << 32 | row*J + j for the valid pairs of segment
// s, grouped by x; segn[s] = the segment's number of valid pairs.
template <bool SG>
__global__ void __launch_bounds__(kLSThreads, 1)
k_sort_local(const uint32_t* __restrict__ pair_x, int64_t npairs,
             const uint32_t* __restrict__ q_row, int J, int log2J,
             unsigned long long* __restrict__ sorted_e, uint32_t* __restrict__ segn) {
    pdl_prologue();
    extern __shared__ __align__(16) uint32_t s_ls[];
    uint32_t* s_key = s_ls;
    uint32_t* s_val = s_ls + kLSSlots;
    __shared__ uint32_t s_warp[33];
    const int tid = threadIdx.x;
#pragma unroll
    for (int k = 0; k < kLSSlotsPer; ++k) {
        s_key[k * kLSThreads + tid] = kEmpty;
        s_val[k * kLSThreads + tid] = 0u;
    }
    const int64_t nseg = (npairs + kLS - 1) / kLS;
    for (int64_t seg = blockIdx.x; seg < nseg; seg += gridDim.x) {
        const int64_t p0 = seg * kLS;
        uint32_t x[kLSPer], e[kLSPer], hr[kLSPer];
#pragma unroll
        for (int i = 0; i < kLSPer; ++i) {
            const int64_t p = p0 + i * kLSThreads + tid;
            x[i] = (p < npairs) ? __ldg(pair_x + p) : kBad;
        }
#pragma unroll
        for (int i = 0; i < kLSPer; ++i) {
            const uint32_t pp = (uint32_t)(p0 + i * kLSThreads + tid);   // npairs < 2^32 here
            const uint32_t q = (log2J >= 0) ? (pp >> log2J) : pp / (uint32_t)J;
            e[i] = pp - q * (uint32_t)J;
            if (x[i] != kBad) {
                e[i] += __ldg(q_row + q) * (uint32_t)J;
                if (SG) {
                    // signed hashing: the sign moves to bit 31 of the entry's low word
                    e[i] |= x[i] & 0x80000000u;
                    x[i] &= 0x7fffffffu;
                }
            }
        }
        __syncthreads();   // the previous segment's table is clear
#pragma unroll
        for (int i = 0; i < kLSPer; ++i)
            hr[i] = (x[i] != kBad) ? local_insert(s_key, s_val, x[i]) : 0u;
        __syncthreads();
        // slot starts: exclusive prefix of the counts in the order (thread,
        // k) over the slots tid + k*kLSThreads that thread tid owns
        uint32_t c[kLSSlotsPer], own = 0u;
#pragma unroll
        for (int k = 0; k < kLSSlotsPer; ++k) {
            c[k] = s_val[k * kLSThreads + tid];
            own += c[k];
        }
        uint32_t total;
        uint32_t run = block_exclusive_scan(own, s_warp, &total);
#pragma unroll
        for (int k = 0; k < kLSSlotsPer; ++k) {
            s_val[k * kLSThreads + tid] = run;
            run += c[k];
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kLSPer; ++i) {
            if (x[i] == kBad) continue;
            const uint32_t pos = s_val[hr[i] & 0xffffu] + (hr[i] >> 16);
            sorted_e[p0 + pos] = ((unsigned long long)x[i] << 32) | e[i];
        }
        if (tid == 0) segn[seg] = total;
        __syncthreads();
#pragma unroll
        for (int k = 0; k < kLSSlotsPer; ++k) {
            s_key[k * kLSThreads + tid] = kEmpty;
            s_val[k * kLSThreads + tid] = 0u;
        }
    }
}

// ---------------------------------------------------------------------------
// Stable LSD radix sort of the pairs by bucket x.
//
// The keys are the bucket indices (at most 32 bits); the sort makes P passes of
// D <= 11 bits each (RadixPlan).  A pass cuts its input into TILES of kRTile
// consecutive entries and takes three kernels:
//   up       each tile's count of every digit, cnt[digit][tile];
//   colscan  for every digit, the exclusive prefix of its counts over the
//            tiles (in place, one warp per digit) and its total; the last CTA
//            to finish turns the totals into the digits' start positions;
//   down     each tile ranks every entry among the tile's entries of the same
//            digit in input order (warp by warp, lane by lane) and stores it at
//              start[digit] + cnt[digit][tile] + rank,
//            staging the tile in shared memory in digit order first, so that
//            the entries of one digit leave the CTA as one contiguous run.
// Entries of equal digit keep their input order, so after the last pass the
// entries are ordered by bucket and, within a bucket, by pair index
// p = q*J + j, whatever the scheduling: the sort is deterministic.  No kernel
// waits for another CTA.  The first pass reads the forward's pair buckets and
// id rows and drops the pairs of bad ids; its colscan writes the number of
// valid pairs to stats[0], which the later passes and the reduce read.
constexpr int kRThreads = 256;
constexpr int kRWarps = kRThreads / 32;
constexpr int kRPer = 32;                        // entries per thread and tile
constexpr int kRWarpKeys = 32 * kRPer;           // entries per warp and tile
constexpr int kRTile = kRThreads * kRPer;        // entries per tile
constexpr int kRMaxDigits = 1 << kRadixMaxBits;
constexpr int kRMaxOwn = kRMaxDigits / kRThreads; // digits per thread at most
static_assert(kRWarpKeys < 65536, "per-warp digit counts are 16-bit");

// Exclusive scan of one value per thread over a CTA of kRThreads threads.
__device__ __forceinline__ uint32_t rblock_exclusive_scan(uint32_t v, uint32_t* s_w,
                                                          uint32_t* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    uint32_t pre = 0, tot = 0;
#pragma unroll
    for (int w = 0; w < kRWarps; ++w) {
        const uint32_t c = s_w[w];
        pre += (w < warp) ? c : 0u;
        tot += c;
    }
    __syncthreads();
    *total = tot;
    return pre + x - v;
}

// Entry of pair p from its bucket x (kBad for a bad id) and its id's output
// row: x << 32 | row*J + j, or ~0 when invalid.  Buckets are below 2^32 - 1,
// so an all-ones entry is never valid.
template <bool SG>
__device__ __forceinline__ unsigned long long radix_pair_entry(uint32_t x, uint32_t row,
                                                               uint32_t p, int J, int log2J) {
    if (x == kBad) return ~0ull;
    const uint32_t q = (log2J >= 0) ? (p >> log2J) : p / (uint32_t)J;
    uint32_t r = row * (uint32_t)J + (p - q * (uint32_t)J);
    if (SG) {
        // signed hashing: the sign moves to bit 31 of the entry's low word
        r |= x & 0x80000000u;
        x &= 0x7fffffffu;
    }
    return ((unsigned long long)x << 32) | r;
}

template <bool FIRST>
__device__ __forceinline__ int64_t radix_count(int64_t npairs,
                                               const unsigned long long* __restrict__ stats) {
    if (FIRST) return npairs;
    const unsigned long long v = stats[0];
    return (int64_t)(v < (unsigned long long)npairs ? v : (unsigned long long)npairs);
}

// up: cnt[d][tile] = entries of the tile with digit d (every tile writes all
// of its nd counts, zeros included).
template <bool FIRST, bool SG>
__global__ void __launch_bounds__(kRThreads)
k_radix_up(const uint32_t* __restrict__ pair_x, const unsigned long long* __restrict__ in_e,
           int64_t npairs, const unsigned long long* __restrict__ stats, int shift, int bits,
           int ntiles, uint32_t* __restrict__ cnt) {
    pdl_prologue();
    __shared__ uint32_t s_c[kRMaxDigits];
    const int nd = 1 << bits;
    const uint32_t dmask = (uint32_t)nd - 1u;
    for (int d = threadIdx.x; d < nd; d += kRThreads) s_c[d] = 0u;
    __syncthreads();
    const int64_t n = radix_count<FIRST>(npairs, stats);
    const int64_t t0 = (int64_t)blockIdx.x * kRTile;
    uint32_t hi[kRPer];
#pragma unroll
    for (int i = 0; i < kRPer; ++i) {
        const int64_t p = t0 + (int64_t)i * kRThreads + threadIdx.x;
        if (FIRST) {
            hi[i] = (p < n) ? __ldg(pair_x + p) : kBad;
            if (SG && hi[i] != kBad) hi[i] &= 0x7fffffffu;
        } else {
            hi[i] = (p < n) ? reinterpret_cast<const uint32_t*>(in_e)[2 * p + 1] : kBad;
        }
    }
#pragma unroll
    for (int i = 0; i < kRPer; ++i)
        if (hi[i] != kBad) atomicAdd(&s_c[(hi[i] >> shift) & dmask], 1u);
    __syncthreads();
    for (int d = threadIdx.x; d < nd; d += kRThreads) cnt[(size_t)d * ntiles + blockIdx.x] = s_c[d];
}

// colscan: one warp per digit d rewrites the row cnt[d][0 .. ntiles) as its
// exclusive prefix (the digit's entries in earlier tiles), 512 tiles per round
// with all of a round's loads in flight; tot[d] = the row's total.  The last
// CTA to finish writes dstart[d] = sum of tot[d'] over d' < d and returns the
// ticket counter to zero; with FIRST it also records the number of valid
// pairs (stats[0]) and clears the distinct-bucket count (stats[1]).
constexpr int kCsPer = 16;   // tiles per lane and round
template <bool FIRST>
__global__ void __launch_bounds__(kRThreads)
k_radix_colscan(uint32_t* __restrict__ cnt, int ntiles, int bits, uint32_t* __restrict__ tot,
                uint32_t* __restrict__ dstart, uint32_t* __restrict__ done,
                unsigned long long* __restrict__ stats) {
    pdl_prologue();
    __shared__ uint32_t s_warp[33];
    __shared__ bool s_last;
    const int nd = 1 << bits;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int d = blockIdx.x * kRWarps + warp;
    if (d < nd) {
        uint32_t* row = cnt + (size_t)d * ntiles;
        uint32_t carry = 0;
        for (int t0 = 0; t0 < ntiles; t0 += 32 * kCsPer) {
            // lane l takes tiles t0 + l*kCsPer .. + kCsPer - 1 (consecutive)
            uint32_t v[kCsPer];
            const int tb = t0 + lane * kCsPer;
#pragma unroll
            for (int i = 0; i < kCsPer; ++i) v[i] = (tb + i < ntiles) ? row[tb + i] : 0u;
            uint32_t mine = 0;
#pragma unroll
            for (int i = 0; i < kCsPer; ++i) mine += v[i];
            uint32_t x = mine;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            uint32_t run = carry + x - mine;
#pragma unroll
            for (int i = 0; i < kCsPer; ++i) {
                if (tb + i < ntiles) row[tb + i] = run;
                run += v[i];
            }
            carry += __shfl_sync(0xffffffffu, x, 31);
        }
        if (lane == 0) tot[d] = carry;
    }
    // the last CTA scans the digit totals
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(done, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // nd <= 2048 digits: 8 per thread
    constexpr int kPer = kRMaxDigits / kRThreads;
    uint32_t v[kPer], mine = 0;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int dd = threadIdx.x * kPer + i;
        v[i] = (dd < nd) ? __ldcg(tot + dd) : 0u;
        mine += v[i];
    }
    uint32_t total;
    uint32_t run = rblock_exclusive_scan(mine, s_warp, &total);
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int dd = threadIdx.x * kPer + i;
        if (dd < nd) dstart[dd] = run;
        run += v[i];
    }
    if (threadIdx.x == 0) {
        *done = 0u;
        if (FIRST) {
            stats[0] = total;
            stats[1] = 0;
        }
    }
}

// Shared memory of the down kernel with 2^bits digits.
__host__ __device__ constexpr size_t radix_down_smem(int nd) {
    return sizeof(unsigned long long) * kRTile + (sizeof(uint16_t) * kRWarps + 8) * (size_t)nd;
}

// down: one tile per CTA (see the section comment).
template <bool FIRST, bool SG>
__global__ void __launch_bounds__(kRThreads, 2)
k_radix_down(const uint32_t* __restrict__ pair_x, const uint32_t* __restrict__ q_row,
             const unsigned long long* __restrict__ in_e, unsigned long long* __restrict__ out_e,
             int64_t npairs, const unsigned long long* __restrict__ stats, int J, int log2J,
             int shift, int bits, int ntiles, const uint32_t* __restrict__ cnt,
             const uint32_t* __restrict__ dstart) {
    pdl_prologue();
    extern __shared__ __align__(16) unsigned char r_smem[];
    const int nd = 1 << bits;
    unsigned long long* s_tile = reinterpret_cast<unsigned long long*>(r_smem);   // [kRTile]
    uint16_t* s_hist = reinterpret_cast<uint16_t*>(s_tile + kRTile);               // [kRWarps][nd]
    uint32_t* s_lst = reinterpret_cast<uint32_t*>(s_hist + kRWarps * nd);          // [nd]
    uint32_t* s_base = s_lst + nd;                                                 // [nd]
    __shared__ uint32_t s_w[kRWarps];
    const uint32_t dmask = (uint32_t)nd - 1u;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t n = radix_count<FIRST>(npairs, stats);
    const int64_t t0 = (int64_t)blockIdx.x * kRTile;
    if (t0 >= n) return;
    {
        uint32_t* z = reinterpret_cast<uint32_t*>(s_hist);
        for (int i = threadIdx.x; i < kRWarps * nd / 2; i += kRThreads) z[i] = 0u;
    }
    // load, warp w taking entries t0 + w*kRWarpKeys + i*32 + lane (i in order)
    unsigned long long e[kRPer];
    {
        const int64_t wb = t0 + (int64_t)warp * kRWarpKeys + lane;
        if (FIRST) {
            // every load is issued before any is used: buckets, then id rows
            uint32_t x[kRPer], row[kRPer];
#pragma unroll
            for (int i = 0; i < kRPer; ++i) {
                const int64_t p = wb + i * 32;
                x[i] = (p < n) ? __ldg(pair_x + p) : kBad;
            }
#pragma unroll
            for (int i = 0; i < kRPer; ++i) {
                const uint32_t pp = (uint32_t)(wb + i * 32);   // npairs < 2^32 here
                const uint32_t q = (log2J >= 0) ? (pp >> log2J) : pp / (uint32_t)J;
                row[i] = (wb + i * 32 < n) ? __ldg(q_row + q) : 0u;
            }
#pragma unroll
            for (int i = 0; i < kRPer; ++i)
                e[i] = radix_pair_entry<SG>(x[i], row[i], (uint32_t)(wb + i * 32), J, log2J);
        } else {
#pragma unroll
            for (int i = 0; i < kRPer; ++i) {
                const int64_t p = wb + i * 32;
                e[i] = (p < n) ? __ldcs(in_e + p) : ~0ull;
            }
        }
    }
    __syncthreads();
    // rank each entry among the warp's entries of its digit, in input order
    uint32_t rank[kRPer];
    {
        uint16_t* hw = s_hist + warp * nd;
        const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
        for (int i = 0; i < kRPer; ++i) {
            const bool valid = e[i] != ~0ull;
            const uint32_t dg = valid ? ((uint32_t)(e[i] >> (32 + shift)) & dmask) : 0xffffffffu;
            const uint32_t peers = __match_any_sync(0xffffffffu, dg);
            const int leader = __ffs(peers) - 1;
            uint32_t base = 0;
            if (valid && lane == leader) {
                base = hw[dg];
                hw[dg] = (uint16_t)(base + __popc(peers));
            }
            base = __shfl_sync(0xffffffffu, base, leader);
            rank[i] = base + __popc(peers & lt);
            __syncwarp();
        }
    }
    __syncthreads();
    // thread t owns digits [t*own, t*own + own) (own = 1 below 256 digits):
    // warp prefixes, the tile's count of each digit, the digits' starts inside
    // the tile, and their bases in the output
    const int own = nd >= kRThreads ? nd / kRThreads : 1;
    const int d0 = threadIdx.x * own;
    const bool owner = d0 < nd;
    uint32_t mine = 0;
    uint32_t cnt_own[kRMaxOwn];
#pragma unroll
    for (int k = 0; k < kRMaxOwn; ++k) {
        cnt_own[k] = 0;
        if (k < own && owner) {
            const int d = d0 + k;
            uint32_t run = 0;
#pragma unroll
            for (int w = 0; w < kRWarps; ++w) {
                const uint32_t c = s_hist[w * nd + d];
                s_hist[w * nd + d] = (uint16_t)run;
                run += c;
            }
            cnt_own[k] = run;
            mine += run;
        }
    }
    uint32_t tile_n;
    uint32_t lst = rblock_exclusive_scan(mine, s_w, &tile_n);
#pragma unroll
    for (int k = 0; k < kRMaxOwn; ++k)
        if (k < own && owner) {
            const int d = d0 + k;
            s_lst[d] = lst;
            s_base[d] = __ldg(dstart + d) + __ldg(cnt + (size_t)d * ntiles + blockIdx.x) - lst;
            lst += cnt_own[k];
        }
    __syncthreads();
    // stage the tile in digit order
#pragma unroll
    for (int i = 0; i < kRPer; ++i) {
        if (e[i] == ~0ull) continue;
        const uint32_t dg = (uint32_t)(e[i] >> (32 + shift)) & dmask;
        s_tile[s_lst[dg] + s_hist[warp * nd + dg] + rank[i]] = e[i];
    }
    __syncthreads();
    // stores in tile order: the entries of one digit are consecutive in both
    for (int l = threadIdx.x; l < (int)tile_n; l += kRThreads) {
        const unsigned long long v = s_tile[l];
        const uint32_t pos = s_base[(uint32_t)(v >> (32 + shift)) & dmask] + (uint32_t)l;
        if ((int64_t)pos < npairs) out_e[pos] = v;   // always, when the counts are consistent
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
               unsigned long long* __restrict__ stats, int64_t npairs,
               const float* __restrict__ gout, int d, int Z, int J, int log2J, int L, int64_t G,
               uint32_t smask, double* __restrict__ g, int log2gs, bool count_runs) {
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

    uint32_t nstart = 0;   // distinct buckets: entries whose bucket differs from the one before
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
        if (count_runs)
            nstart += (e0 == 0 || (uint32_t)(__ldg(sorted_e + e0 - 1) >> 32) != cur) ? 1u : 0u;
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
            // does (entries in bucket order)
            if (xs[kRU - 1] == cur) {
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
                        ++nstart;
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
    if (count_runs && lg == 0 && nstart) atomicAdd(stats + 1, (unsigned long long)nstart);
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

// (at most 64 registers for KE <= 2: 4 CTAs per SM; at 72 registers, 3 per
// SM, the paper micro-benchmark shape with Z = 64 reduced in 0.085 ms
// against 0.073 ms with the bound)
template <int KE, bool ZDIV, bool JPOW2>
__global__ void __launch_bounds__(kThreads, (KE <= 2) ? 4 : 1)
k_warp_range_reduce(const unsigned long long* __restrict__ sorted_e,
                    unsigned long long* __restrict__ stats, int64_t npairs,
                    const float* __restrict__ gout, int d, int Z, int J, int log2J, int L,
                    int64_t G, uint32_t smask, double* __restrict__ g, bool count_runs) {
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
    uint32_t nstart = 0;   // distinct buckets: entries whose bucket differs from the one before
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
        if (count_runs)
            nstart += (e0 == 0 || (uint32_t)(__ldg(sorted_e + e0 - 1) >> 32) != cur) ? 1u : 0u;
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
            if (xs[kWU - 1] == cur) {
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
                        ++nstart;
                    }
#pragma unroll
                    for (int k = 0; k < KE; ++k) kahan_add(s[k], c[k], v[u][k]);
                }
            }
        }
        flush(cur);
        __syncwarp();
    }
    if (count_runs && lane == 0 && nstart) atomicAdd(stats + 1, (unsigned long long)nstart);
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

// L2 policy for data read once (the upstream gradient, the sorted entries):
// evicted first, so that the streams do not push the fp64 accumulator and the
// shared array out of L2.
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, uint64_t pol) {
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2;\n"
                 :: "r"(sa), "l"(gmem), "l"(pol) : "memory");
}
__device__ __forceinline__ unsigned long long ld_once_u64(const unsigned long long* p,
                                                          uint64_t pol) {
    unsigned long long v;
    asm volatile("ld.global.nc.L2::cache_hint.u64 %0, [%1], %2;" : "=l"(v) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" :: "n"(N) : "memory");
}

// Where the staged reduce puts each run's sum (SINK):
//   kSinkF64   added into the fp64 gradient accumulator g (red.global.add.f64);
//   kSinkOnce  added into the task's ELEMENT WINDOW: the runs of a task come in
//              ascending bucket order, so the 32 elements [wb, wb + 32) that
//              lane z holds (element wb + z) slide forward; an element that
//              leaves the window has all of the task's contributions.  If no
//              other task can add to it (no bucket of the task before or after
//              this one reaches it), its gradient is final and is stored once
//              into ws.gexp (fp32).  Otherwise its partial sum goes to the
//              task's boundary record (bnd[task][0..32): the window of its
//              first bucket, [32..64): of its last), and k_window_combine
//              stores it.  Every element's additions then happen in a fixed
//              order, and nothing is added atomically.
constexpr int kSinkF64 = 0;
constexpr int kSinkOnce = 1;

template <int SINK>
__global__ void __launch_bounds__(kThreads, 4)
k_async_reduce(const unsigned long long* __restrict__ sorted_e,
               unsigned long long* __restrict__ stats, int64_t npairs,
               const float* __restrict__ gout, int64_t G, uint32_t smask,
               double* __restrict__ g, WindowSink ws, const uint32_t* __restrict__ segn,
               bool count_runs) {
    pdl_prologue();
    __shared__ __align__(16) float s_ring[kWarps][kAD][kAS][32];
    __shared__ unsigned long long s_ent[kWarps][kAPiece];
    // segn: the segment-local layout (k_sort_local), kLS / kAPiece tasks per
    // segment, each cut at the segment's valid entries; otherwise one sorted
    // run of stats[0] valid entries
    constexpr int kPieces = kLS / kAPiece;
    const bool local = segn != nullptr;
    const int64_t total =
        local ? npairs : (int64_t)(stats[0] < (unsigned long long)npairs ? stats[0] : npairs);
    const int64_t ntasks =
        local ? ((npairs + kLS - 1) / kLS) * kPieces : (total + kAPiece - 1) / kAPiece;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    unsigned long long* ent = s_ent[warp];
    const int64_t wstride = (int64_t)gridDim.x * kWarps;
    constexpr unsigned long long kNone = (unsigned long long)kBad << 32;
    const uint64_t pol = l2_evict_first();
    float sum = 0.f, comp = 0.f;
    // window sink: lane z holds element wb + z; the task's head boundary ends
    // at hb_end, its tail boundary starts at tb_start; hx and tx are the first
    // elements of its first and last buckets
    int64_t wb = 0, hb_end = 0, tb_start = 0, hx = 0, tx = 0, task = 0;
    float acc = 0.f, accc = 0.f;
    auto finalize = [&](int lim) {   // the window's first lim elements are done
        if (lane < lim) {
            const int64_t e = wb + lane;
            const float v = acc - accc;
            if (e < hb_end || e >= tb_start) {
                float* rec = ws.bnd + task * 64;
                if (e < hx + 32) rec[e - hx] = v;
                else rec[32 + (e - tx)] = v;
            } else if (v != 0.f) {
                ws.gexp[e] = v;
            }
        }
    };
    auto flush = [&](uint32_t x) {
        if (SINK == kSinkF64) {
            if (sum != 0.f) red_add_f64(g + (int64_t)x * G + lane, widen(sum));
        } else {
            const int64_t xb = (int64_t)x * G;
            const int64_t sh = xb - wb;           // >= 0: buckets ascend
            if (sh > 0) {
                finalize(sh < 32 ? (int)sh : 32);
                if (sh >= 32) {
                    acc = accc = 0.f;
                } else {
                    const float a2 = __shfl_down_sync(0xffffffffu, acc, (int)sh);
                    const float c2 = __shfl_down_sync(0xffffffffu, accc, (int)sh);
                    const bool in = lane + (int)sh < 32;
                    acc = in ? a2 : 0.f;
                    accc = in ? c2 : 0.f;
                }
                wb = xb;
            }
            kahan_add(acc, accc, sum - comp);
        }
        sum = comp = 0.f;
    };
    uint32_t nstart = 0;   // distinct buckets: entries whose bucket differs from the one before
    for (int64_t t = (int64_t)blockIdx.x * kWarps + warp; t < ntasks; t += wstride) {
        int64_t e0;
        int n;
        if (local) {
            const int64_t s = t / kPieces;
            const int k = (int)(t - s * kPieces);
            const int left = (int)__ldg(segn + s) - k * kAPiece;
            if (left <= 0) continue;
            e0 = s * kLS + (int64_t)k * kAPiece;
            n = left < kAPiece ? left : kAPiece;
        } else {
            e0 = t * kAPiece;
            n = (int)((e0 + kAPiece < total) ? kAPiece : total - e0);
        }
#pragma unroll
        for (int h = 0; h < kAPiece; h += 32)
            ent[h + lane] = (h + lane < n) ? ld_once_u64(sorted_e + e0 + h + lane, pol) : kNone;
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
                                   gout + (uint64_t)r * 32u + (uint32_t)(part * 4), pol);
                    }
                }
            }
            cp_async_commit();
        };
#pragma unroll
        for (int st = 0; st < kAD - 1; ++st) issue(st);
        sum = comp = 0.f;
        uint32_t cur = (uint32_t)(ent[0] >> 32);
        // the previous entry's bucket: the window's head boundary, and the count
        // of distinct buckets when this pass makes it
        const bool need_prev = (SINK != kSinkF64) || count_runs;
        const uint32_t xprev = (e0 > 0 && !local && need_prev)
                                   ? (uint32_t)(__ldg(sorted_e + e0 - 1) >> 32)
                                   : kBad;
        nstart += (e0 == 0 || xprev != cur) ? 1u : 0u;
        if (SINK != kSinkF64) {
            task = t;
            hx = (int64_t)cur * G;
            tx = (int64_t)(uint32_t)(ent[n - 1] >> 32) * G;
            hb_end = (e0 > 0) ? (int64_t)xprev * G + 32 : 0;
            tb_start = (e0 + n < total) ? (int64_t)(uint32_t)(__ldg(sorted_e + e0 + n) >> 32) * G
                                        : INT64_MAX;
            wb = hx;
            acc = accc = 0.f;
        }
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
            if (xlast == cur) {
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
                        ++nstart;
                    }
                    kahan_add(sum, comp, v[i]);
                }
            }
            __syncwarp();
        }
        flush(cur);
        if (SINK != kSinkF64) finalize(32);
        cp_async_wait<0>();
        __syncwarp();
    }
    // (the local layout's runs are per segment: no distinct-bucket count)
    if (count_runs && lane == 0 && nstart && !local) atomicAdd(stats + 1, (unsigned long long)nstart);
}

// The boundary elements of the window reduce.  Between task j - 1 and task j
// the elements [G*x_first(j), G*x_last(j-1) + 32) got partial sums from both
// (and from more tasks when one bucket fills several).  One warp per task
// boundary j, lane z on element e = G*x_first(j) + z: if e lies there and not
// also past the next boundary, this warp owns e.  The tasks that hold e are
// j, j - 1, ... down to the first that does not: the warp loads the bounds of
// 32 tasks at a time (one per lane), each lane counts its tasks from them,
// then loads their partials with independent loads and adds them in task
// order (j first) in fp64, and stores the sum into ws.gexp.
__global__ void __launch_bounds__(kThreads)
k_window_combine(const unsigned long long* __restrict__ sorted_e,
                 const unsigned long long* __restrict__ stats, int64_t npairs, int64_t G,
                 WindowSink ws) {
    pdl_prologue();
    const int64_t total = (int64_t)(stats[0] < (unsigned long long)npairs ? stats[0] : npairs);
    const int64_t ntasks = (total + kAPiece - 1) / kAPiece;
    const int lane = threadIdx.x & 31;
    auto xat = [&](int64_t i) { return (int64_t)(uint32_t)(__ldg(sorted_e + i) >> 32) * G; };
    auto xlast = [&](int64_t k) {
        return xat(((k + 1) * kAPiece < total ? (k + 1) * kAPiece : total) - 1);
    };
    for (int64_t j = 1 + (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5); j < ntasks;
         j += (int64_t)gridDim.x * kWarps) {
        const int64_t xfj = xat(j * kAPiece);
        const int64_t xlp = xat(j * kAPiece - 1);
        const int64_t xfn = (j + 1 < ntasks) ? xat((j + 1) * kAPiece) : INT64_MAX;
        const int64_t e = xfj + lane;
        // shared with task j - 1, and no later boundary owns it
        bool open = e < xlp + 32 && e < xfn;
        if (!__any_sync(0xffffffffu, open)) continue;
        double tot = 0.0;
        for (int64_t kb = j; kb >= 0 && __any_sync(0xffffffffu, open); kb -= 32) {
            // lane i: bounds of task kb - i
            const int64_t kl = kb - lane;
            const int64_t xfk = (kl >= 0) ? xat(kl * kAPiece) : INT64_MAX;
            const int64_t xlk = (kl >= 0) ? xlast(kl) : 0;
            // tasks kb, kb - 1, ... holding e: the first ncnt of this round
            int ncnt = 0;
            for (int i = 0; i < 32; ++i) {
                // (most boundaries are shared by two tasks only)
                if (!__any_sync(0xffffffffu, open)) break;
                const int64_t xf = __shfl_sync(0xffffffffu, xfk, i);
                const int64_t xl = __shfl_sync(0xffffffffu, xlk, i);
                const bool holds = open && e >= xf && e < xl + 32 && (e < xf + 32 || e >= xl);
                if (holds) ++ncnt;
                else open = false;
            }
            // their partials, loaded independently, added in task order
            for (int i0 = 0; i0 < 32; i0 += 8) {
                if (!__any_sync(0xffffffffu, i0 < ncnt)) break;
                float p[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = i0 + u;
                    const int64_t xf = __shfl_sync(0xffffffffu, xfk, i);
                    const int64_t xl = __shfl_sync(0xffffffffu, xlk, i);
                    p[u] = 0.f;
                    if (i < ncnt) {
                        const float* rec = ws.bnd + (kb - i) * 64;
                        p[u] = (e < xf + 32) ? rec[e - xf] : rec[32 + (e - xl)];
                    }
                }
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (i0 + u < ncnt) tot += widen(p[u]);
            }
        }
        const float v = narrow(tot);
        if (v != 0.f && e < xlp + 32 && e < xfn) ws.gexp[e] = v;
    }
}

template <int KE, bool ZDIV, bool JPOW2>
cudaError_t warp_reduce_launch(const SortedBuffers& sb, int64_t npairs, const float* gout,
                               const DevParams& p, double* g, int log2J, bool count_runs,
                               int sm_count, cudaStream_t st) {
    const int64_t ntasks = (npairs + kPiece - 1) / kPiece;   // upper bound
    const int grid = grid_for(k_warp_range_reduce<KE, ZDIV, JPOW2>, sm_count,
                              (ntasks + kWarps - 1) / kWarps);
    return launch_k(k_warp_range_reduce<KE, ZDIV, JPOW2>, dim3(grid), dim3(kThreads), 0, st,
                    sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, log2J, p.L, p.G, p.smask, g,
                    count_runs);
}

template <int KE>
cudaError_t warp_reduce_inst(const SortedBuffers& sb, int64_t npairs, const float* gout,
                             const DevParams& p, double* g, bool count_runs, int sm_count,
                             cudaStream_t st) {
    const int log2J = (p.J & (p.J - 1)) == 0 ? ceil_log2(p.J) : -1;
    if (p.d % p.Z == 0)
        return warp_reduce_launch<KE, true, true>(sb, npairs, gout, p, g, 0, count_runs, sm_count,
                                                  st);
    if (log2J >= 0)
        return warp_reduce_launch<KE, false, true>(sb, npairs, gout, p, g, log2J, count_runs,
                                                   sm_count, st);
    return warp_reduce_launch<KE, false, false>(sb, npairs, gout, p, g, 0, count_runs, sm_count,
                                                st);
}

template <int VW, int KC, bool JPOW2, bool ZDIV>
cudaError_t reduce_launch(const SortedBuffers& sb, int64_t npairs, const float* gout,
                          const DevParams& p, double* g, int log2J, int log2gs, bool count_runs,
                          int sm_count, cudaStream_t st) {
    const int gpc = kWarps * (32 >> log2gs);
    const size_t smem = sizeof(float) * (size_t)gpc * (size_t)p.L;
    const int64_t ntasks = (npairs + kPiece - 1) / kPiece;   // upper bound
    const int64_t work_blocks = (ntasks + gpc - 1) / gpc;
    const int grid = grid_for(k_range_reduce<VW, KC, JPOW2, ZDIV>, sm_count, work_blocks, smem);
    return launch_k(k_range_reduce<VW, KC, JPOW2, ZDIV>, dim3(grid), dim3(kThreads), smem, st,
                    sb.sorted_e, sb.stats, npairs, gout, p.d, p.Z, p.J, log2J, p.L, p.G, p.smask, g, log2gs,
                    count_runs);
}

template <int VW, int KC>
cudaError_t reduce_inst(const SortedBuffers& sb, int64_t npairs, const float* gout,
                        const DevParams& p, double* g, int log2gs, bool count_runs, int sm_count,
                        cudaStream_t st) {
    const int log2J = (p.J & (p.J - 1)) == 0 ? ceil_log2(p.J) : -1;
    if (p.d % p.Z == 0)
        return reduce_launch<VW, KC, true, true>(sb, npairs, gout, p, g, 0, log2gs, count_runs,
                                                 sm_count, st);
    if (log2J >= 0)
        return reduce_launch<VW, KC, true, false>(sb, npairs, gout, p, g, log2J, log2gs,
                                                  count_runs, sm_count, st);
    return reduce_launch<VW, KC, false, false>(sb, npairs, gout, p, g, 0, log2gs, count_runs,
                                               sm_count, st);
}

}  // namespace

RadixPlan radix_plan(uint64_t R, int digit_bits) {
    // buckets lie in [0, R - 1]: nbits bits with 2^nbits >= R
    int nbits = 1;
    while (nbits < 32 && (uint64_t(1) << nbits) < R) ++nbits;
    const int dmax = digit_bits > 0 ? digit_bits : kRadixMaxBits;
    RadixPlan pl{};
    pl.passes = (nbits + dmax - 1) / dmax;
    const int D = digit_bits > 0 ? digit_bits : (nbits + pl.passes - 1) / pl.passes;
    for (int k = 0; k < pl.passes; ++k) {
        pl.shift[k] = k * D;
        pl.bits[k] = (nbits - k * D) < D ? (nbits - k * D) : D;
    }
    return pl;
}

int64_t radix_tiles(int64_t npairs) {
    const int64_t t = (npairs + kRTile - 1) / kRTile;
    return t < 1 ? 1 : t;
}

template <bool FIRST, bool SG>
cudaError_t radix_pass(const SortedBuffers& sb, const unsigned long long* in,
                       unsigned long long* out, int64_t npairs, int J, int log2J,
                       const RadixPlan& plan, int k, cudaStream_t st) {
    const int ntiles = (int)radix_tiles(npairs);
    const int bits = plan.bits[k], shift = plan.shift[k];
    const int nd = 1 << bits;
    cudaError_t e = launch_k(k_radix_up<FIRST, SG>, dim3(ntiles), dim3(kRThreads), 0, st,
                             sb.pair_x, in, npairs, sb.stats, shift, bits, ntiles, sb.cnt);
    if (e != cudaSuccess) return e;
    e = launch_k(k_radix_colscan<FIRST>, dim3((nd + kRWarps - 1) / kRWarps), dim3(kRThreads), 0,
                 st, sb.cnt, ntiles, bits, sb.tot, sb.dstart, sb.done, sb.stats);
    if (e != cudaSuccess) return e;
    const size_t smem = radix_down_smem(nd);
    e = cudaFuncSetAttribute(k_radix_down<FIRST, SG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    return launch_k(k_radix_down<FIRST, SG>, dim3(ntiles), dim3(kRThreads), smem, st, sb.pair_x,
                    sb.q_row, in, out, npairs, sb.stats, J, log2J, shift, bits, ntiles, sb.cnt,
                    sb.dstart);
}

cudaError_t launch_radix_sort(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                              const RadixPlan& plan, cudaStream_t st) {
    const int log2J = (J & (J - 1)) == 0 ? ceil_log2(J) : -1;
    const unsigned long long* in = nullptr;
    for (int k = 0; k < plan.passes; ++k) {
        // the last pass writes sorted_e; earlier ones alternate with tmp_e
        unsigned long long* out = ((plan.passes - 1 - k) % 2 == 0) ? sb.sorted_e : sb.tmp_e;
        cudaError_t e;
        if (k == 0)
            e = smask ? radix_pass<true, true>(sb, in, out, npairs, J, log2J, plan, k, st)
                      : radix_pass<true, false>(sb, in, out, npairs, J, log2J, plan, k, st);
        else
            e = radix_pass<false, false>(sb, in, out, npairs, J, log2J, plan, k, st);
        if (e != cudaSuccess) return e;
        in = out;
    }
    return cudaSuccess;
}

int64_t sorted_scan_blocks(int64_t R) { return (R + kScanChunk - 1) / kScanChunk; }

cudaError_t launch_sorted_scan(const SortedBuffers& sb, int64_t R, const Touched* touched,
                               cudaStream_t st) {
    const int64_t nblk = sorted_scan_blocks(R);
    const Touched tc = touched ? *touched : Touched{};
    cudaError_t e = launch_k(k_scan_reduce, dim3((unsigned)nblk), dim3(kScanThreads), 0, st,
                             sb.ccnt, R, sb.bsum, sb.bnz);
    if (e != cudaSuccess) return e;
    return launch_k(k_scan_apply, dim3((unsigned)nblk), dim3(kScanThreads), 0, st, sb.ccnt, R,
                    sb.bsum, sb.bnz, sb.start, tc, sb.stats);
}

cudaError_t launch_sorted_scatter(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                                  int sm_count, cudaStream_t st) {
    const int log2J = (J & (J - 1)) == 0 ? ceil_log2(J) : -1;
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    if (smask) {
        const int grid = grid_for(k_sort_scatter<true>, sm_count, nseg);
        return launch_k(k_sort_scatter<true>, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x,
                        npairs, sb.q_row, J, log2J, sb.start, sb.sorted_e);
    }
    const int grid = grid_for(k_sort_scatter<false>, sm_count, nseg);
    return launch_k(k_sort_scatter<false>, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x, npairs,
                    sb.q_row, J, log2J, sb.start, sb.sorted_e);
}

cudaError_t launch_sorted_count(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                                int sm_count, cudaStream_t st) {
    const int64_t nseg = (npairs + kSeg - 1) / kSeg;
    const int grid = grid_for(k_sort_count, sm_count, nseg);
    return launch_k(k_sort_count, dim3(grid), dim3(kSegThreads), 0, st, sb.pair_x, npairs, smask,
                    sb.ccnt);
}

cudaError_t launch_mark_pairs(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                              const Touched& touched, int sm_count, cudaStream_t st) {
    const int64_t chunks = (npairs + kMarkChunk - 1) / kMarkChunk;
    const int grid = grid_for(k_mark_pairs, sm_count, chunks);
    return launch_k(k_mark_pairs, dim3(grid), dim3(kThreads), 0, st, sb.pair_x, npairs, smask,
                    touched);
}

bool window_reduce_ok(const DevParams& p, const float* gout) {
    return p.Z == 32 && p.d % 32 == 0 && (((uintptr_t)gout & 15u) == 0);
}

int64_t window_records(int64_t npairs) { return (npairs + kAPiece - 1) / kAPiece; }

cudaError_t launch_window_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, const WindowSink& ws, int sm_count,
                                 cudaStream_t st) {
    if (!window_reduce_ok(p, gout)) return cudaErrorInvalidValue;
    const int64_t ntasks = window_records(npairs);   // upper bound
    const int64_t blocks = (ntasks + kWarps - 1) / kWarps;
    int grid = grid_for(k_async_reduce<kSinkOnce>, sm_count, blocks);
    cudaError_t e = launch_k(k_async_reduce<kSinkOnce>, dim3(grid), dim3(kThreads), 0, st,
                             sb.sorted_e, sb.stats, npairs, gout, p.G, p.smask,
                             (double*)nullptr, ws, (const uint32_t*)nullptr, true);
    if (e != cudaSuccess) return e;
    grid = grid_for(k_window_combine, sm_count, blocks);
    return launch_k(k_window_combine, dim3(grid), dim3(kThreads), 0, st, sb.sorted_e,
                    (const unsigned long long*)sb.stats, npairs, p.G, ws);
}

int64_t local_segments(int64_t npairs) { return (npairs + kLS - 1) / kLS; }

bool local_sort_ok(const DevParams& p, const float* gout) { return window_reduce_ok(p, gout); }

cudaError_t launch_sort_local(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                              int sm_count, cudaStream_t st) {
    if (npairs <= 0) return cudaSuccess;
    const int log2J = ((J & (J - 1)) == 0) ? ceil_log2(J) : -1;
    const size_t smem = sizeof(uint32_t) * 2 * (size_t)kLSSlots;
    auto kern = smask ? k_sort_local<true> : k_sort_local<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kLSThreads, smem) !=
            cudaSuccess || per_sm < 1)
        per_sm = 1;
    const int64_t nseg = local_segments(npairs);
    const int grid = (int)(nseg < (int64_t)sm_count * per_sm ? nseg : (int64_t)sm_count * per_sm);
    return launch_k(kern, dim3(grid), dim3(kLSThreads), smem, st, sb.pair_x, npairs, sb.q_row, J,
                    log2J, sb.sorted_e, sb.segn);
}

cudaError_t launch_sorted_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, double* g, bool local, bool count_runs,
                                 int sm_count, cudaStream_t st) {
    if (local && !window_reduce_ok(p, gout)) return cudaErrorInvalidValue;
    // 32-element chunks tiling the rows: asynchronous shared-memory staging
    if (window_reduce_ok(p, gout)) {
        // 3 CTAs per SM (measured at the Criteo-TB shape: 0.170 ms against
        // 0.177 with 4, the occupancy limit, 0.199 with 2 and 0.197 with 6):
        // fewer random gathers in flight keep the DRAM more efficient
        const int64_t ntasks = (npairs + kAPiece - 1) / kAPiece;   // upper bound
        int grid = grid_for(k_async_reduce<kSinkF64>, sm_count, (ntasks + kWarps - 1) / kWarps);
        if (grid > 3 * sm_count) grid = 3 * sm_count;
        return launch_k(k_async_reduce<kSinkF64>, dim3(grid), dim3(kThreads), 0, st, sb.sorted_e,
                        sb.stats, npairs, gout, p.G, p.smask, g, WindowSink{},
                        local ? (const uint32_t*)sb.segn : (const uint32_t*)nullptr, count_runs);
    }
    // blocks of 32+ elements: one warp per task, one element per lane
    if (p.L >= 32) {
        if (p.L <= 32) return warp_reduce_inst<1>(sb, npairs, gout, p, g, count_runs, sm_count, st);
        if (p.L <= 64) return warp_reduce_inst<2>(sb, npairs, gout, p, g, count_runs, sm_count, st);
        if (p.L <= 128)
            return warp_reduce_inst<4>(sb, npairs, gout, p, g, count_runs, sm_count, st);
    }
    const bool vec = (p.Z % 4 == 0) && (p.d % 4 == 0) && (((uintptr_t)gout & 15u) == 0);
    const int vw = vec ? 4 : 1;
    const int V = (p.L + vw - 1) / vw;
    const int log2gs = V <= 32 ? ceil_log2(V) : 5;
    const int kc = V <= 32 ? 1 : (1 << ceil_log2((V + 31) / 32));
#define PSS_RD(VW, KC) \
    return reduce_inst<VW, KC>(sb, npairs, gout, p, g, log2gs, count_runs, sm_count, st)
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
