// Internal declarations shared by the CUDA translation units of libpss.so.
// Nothing here is part of the public ABI (include/pss.h is).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace pss {

// Hash and shape parameters as the kernels see them.
//   bucket x = ((A*key + B0) mod P) mod R,  P = 2^61 - 1,  loc = G*x
//   Rinv = floor((2^64 - 1) / R) drives the exact "mod R" reduction.
struct DevParams {
    uint64_t A, B0, R, Rinv;
    int64_t G, M;
    int32_t T, d, Z, J, L;
    const int64_t* cards;   // device, T entries
    uint64_t A2, B2;        // sign hash
    uint32_t smask;         // 0x80000000 with signed hashing, else 0 (see pss_device.cuh)
};

// Hash parameters of a seed (host side, shared by pss_create and
// pss_grad_noalloc): s1..s4 are the first four splitmix64 outputs (Steele, Lea
// & Flood 2014) of `seed`, A = 1 + s1 mod (P-1), B0 = s2 mod P for the
// location hash and A2 = 1 + s3 mod (P-1), B2 = s4 mod P for the sign hash.
inline void hash_params_from_seed(uint64_t seed, DevParams* p) {
    const uint64_t p61 = (uint64_t(1) << 61) - 1;
    uint64_t s = seed;
    uint64_t out[4];
    for (int k = 0; k < 4; ++k) {
        s += 0x9e3779b97f4a7c15ULL;
        uint64_t z = s;
        z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
        z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
        out[k] = z ^ (z >> 31);
    }
    p->A = 1 + out[0] % (p61 - 1);
    p->B0 = out[1] % p61;
    p->A2 = 1 + out[2] % (p61 - 1);
    p->B2 = out[3] % p61;
}

// Device error word: smallest id position seen out of range, and flag bits.
struct DevError {
    unsigned long long first_bad;   // ULLONG_MAX when clear
    unsigned int flags;             // kErrOffsets
    unsigned int pad;
};
constexpr unsigned int kErrOffsets = 1u;

// Lane layout of one bag row: VW-wide columns, groups of gs lanes per bag.
struct RowLayout {
    int vw;        // 4 (float4 columns) or 1
    int kc;        // columns per lane
    int log2gs;    // log2(lanes per bag group)
};
RowLayout choose_layout(int d, int Z, int64_t G);

// Touched-block bookkeeping for the sparse optimizer pass.
struct Touched {
    uint32_t* bitmap;                 // R bits
    int64_t* list;                    // bucket indices x, capacity cap
    unsigned long long* count;        // number of entries in list
    int64_t cap;
};

// Radix sort of the sorted backward path: `passes` digits of `bits[k]` bits
// starting at bit shift[k] of the bucket index.
constexpr int kRadixMaxBits = 11;          // digit bits per pass (at most 2048 digits)
constexpr int kRadixMaxPasses = 8;         // 32-bit buckets with 4-bit digits
struct RadixPlan {
    int passes;
    int bits[kRadixMaxPasses];
    int shift[kRadixMaxPasses];
};
// Plan for buckets in [0, R): digit_bits 0 picks at most kRadixMaxBits bits per
// pass, as few passes as that allows, split evenly; 4 .. 11 forces that many.
RadixPlan radix_plan(uint64_t R, int digit_bits);
int64_t radix_tiles(int64_t npairs);   // tiles of one pass

// Buffers of the sorted backward path (see pss_sorted.cu).
struct SortedBuffers {
    uint32_t* pair_x;             // nnz*J buckets written by the forward (0xffffffff: bad id)
    uint32_t* q_row;              // nnz output rows b*T + t written by the forward
    unsigned long long* sorted_e; // nnz*J entries (x << 32 | row*J + j), grouped by x
    unsigned long long* stats;    // [0] valid pairs, [1] distinct buckets
    float* bnd;                   // window reduce: boundary records, 64 floats per task
    uint32_t* segn;               // local sort: valid pairs of each segment
    // counting sort (R <= kCountSortMaxR)
    uint32_t* ccnt;               // R counts per bucket (zero between sorts)
    uint32_t* start;              // R + 1 bucket starts
    uint32_t* bsum;               // per scan chunk: entries
    uint32_t* bnz;                // per scan chunk: non-empty buckets
    // radix sort
    unsigned long long* tmp_e;    // nnz*J entries: the other buffer of the radix passes
    uint32_t* cnt;                // [2^bits][radix_tiles(nnz*J)] per-tile digit counts
    uint32_t* tot;                // [2^kRadixMaxBits] digit totals of the current pass
    uint32_t* dstart;             // [2^kRadixMaxBits] digit start positions of the current pass
    uint32_t* done;               // finished-CTA counter of the column scan (zero between passes)
};
// The counting sort keeps one counter per bucket: it serves R up to this.
constexpr int64_t kCountSortMaxR = int64_t(1) << 22;
int64_t sorted_scan_blocks(int64_t R);
// Counting sort: per-bucket counts of the valid pairs (ccnt must be zero on
// entry), their scan into the bucket starts (which returns ccnt to zero; with
// `touched`, also the list / bitmap of non-empty buckets), and the slot
// scatter into sorted_e (which advances each start to its bucket's end).
cudaError_t launch_sorted_count(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                                int sm_count, cudaStream_t st);
cudaError_t launch_sorted_scan(const SortedBuffers& sb, int64_t R, const Touched* touched,
                               cudaStream_t st);
cudaError_t launch_sorted_scatter(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                                  int sm_count, cudaStream_t st);
// Stable radix sort of the forward's pairs by bucket into sorted_e (three
// kernels per pass; see pss_sorted.cu): entries of one bucket in pair order.
cudaError_t launch_radix_sort(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                              const RadixPlan& plan, cudaStream_t st);
// Touched bitmap / list of the buckets of the forward's pairs.
cudaError_t launch_mark_pairs(const SortedBuffers& sb, int64_t npairs, uint32_t smask,
                              const Touched& touched, int sm_count, cudaStream_t st);
// Segment-local sort (see pss_sorted.cu): the valid entries of each segment of
// consecutive pairs grouped by bucket inside the segment's range of sorted_e,
// their number in segn[local_segments(npairs)].  Serves the shapes of the
// staged reduce (local_sort_ok) with R < 2^32 - 1; any R, no per-bucket state.
int64_t local_segments(int64_t npairs);
bool local_sort_ok(const DevParams& p, const float* gout);
cudaError_t launch_sort_local(const SortedBuffers& sb, int64_t npairs, int J, uint32_t smask,
                              int sm_count, cudaStream_t st);
// Reduce of the sorted entries into g (fp64).  `local`: the entries come from
// the segment-local sort (one run per bucket and segment).  `count_runs`: the
// reduce counts the distinct buckets into stats[1] (the radix sort's entries;
// the counting sort's scan counts them itself).
cudaError_t launch_sorted_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, double* g, bool local, bool count_runs,
                                 int sm_count, cudaStream_t st);
// Window reduce (see pss_sorted.cu): run sums go into each task's sliding
// element window; every element's gradient is stored once into gexp (fp32,
// zero where the batch adds nothing; the caller zero-fills it), in a fixed
// order of additions.  Serves 32-element chunks tiling the rows (Z = 32,
// d % 32 == 0, 16-byte aligned upstream gradient) when the array does not
// wrap.
struct WindowSink {
    float* gexp;    // gradient out, M elements
    float* bnd;     // window_records(npairs) records of 64 floats
};
bool window_reduce_ok(const DevParams& p, const float* gout);
int64_t window_records(int64_t npairs);
cudaError_t launch_window_reduce(const SortedBuffers& sb, int64_t npairs, const float* gout,
                                 const DevParams& p, const WindowSink& ws, int sm_count,
                                 cudaStream_t st);

// Kernel launchers (return the CUDA launch error).  `grid_cap` bounds the
// grid of grid-stride kernels; 0 lets the launcher decide.
cudaError_t launch_locations(const DevParams& p, const int64_t* idx, int64_t nnz,
                             const int64_t* off, int64_t B, int64_t* locs, DevError* err,
                             int sm_count, cudaStream_t st);
// Forward of the bags of batch rows [b_lo, b_hi) of every table (0 <= b_lo <
// b_hi <= B; out, idx and off are the whole batch's); when pair_x / q_row are
// given it also writes those bags' pairs' buckets and ids' output rows for the
// sorted backward path.
cudaError_t launch_forward(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* w, float* out,
                           DevError* err, uint32_t* pair_x, uint32_t* q_row, int64_t b_lo,
                           int64_t b_hi, int sm_count, cudaStream_t st);
// Backward scatter into an fp32 target (scale applied to grad_out) or into an
// fp64 accumulator (scale 1).
cudaError_t launch_scatter(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                           float scale, float* target, const Touched* touched, DevError* err,
                           int sm_count, cudaStream_t st);
cudaError_t launch_scatter64(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                             int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                             double* target, const Touched* touched, DevError* err, int sm_count,
                             cudaStream_t st);
// Optimizer passes: dense over M, or over the touched blocks (one warp per
// distinct block start); g is returned to zero.
cudaError_t launch_update_dense(bool adagrad, float* w, float* Gacc, float* g, int64_t M,
                                float lr, float eps, int sm_count, cudaStream_t st);
cudaError_t launch_update_dense64(bool adagrad, float* w, float* Gacc, double* g, int64_t M,
                                  float lr, float eps, int sm_count, cudaStream_t st);
cudaError_t launch_update_touched(bool adagrad, float* w, float* Gacc, float* g,
                                  const Touched& touched, int64_t G, int32_t L, float lr,
                                  float eps, int sm_count, cudaStream_t st);
cudaError_t launch_update_touched64(bool adagrad, float* w, float* Gacc, double* g,
                                    const Touched& touched, int64_t G, int32_t L, float lr,
                                    float eps, int sm_count, cudaStream_t st);
// out[e] = fp32(g[e]); g[e] = 0 for all e < M.
cudaError_t launch_grad_export(double* g, float* out, int64_t M, int sm_count, cudaStream_t st);
// Clears the bitmap words of the listed starts and resets the list count.
cudaError_t launch_touched_clear(const Touched& touched, int sm_count, cudaStream_t st);
// Circular array: g[z] += g[M + z], g[M + z] = 0 for z < L (g64 or g32).
cudaError_t launch_fold_tail(double* g64, float* g32, int64_t M, int L, cudaStream_t st);
// direction 0: fp32 -> fp64 (widen); 1: fp64 -> fp32 (narrow), n values.
cudaError_t launch_convert(int direction, const void* in, void* out, int64_t n, int sm_count,
                           cudaStream_t st);

}  // namespace pss
