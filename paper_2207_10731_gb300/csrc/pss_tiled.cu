// Tiled forward (hash + gather + sum-pool) and backward scatter kernels.
//
// The forward gives each warp its own tile (see k_forward_warp).  The atomic
// backward scatter gives each CTA a TILE of `tb` consecutive bags of one table
// (bag slots t*B + b0 .. t*B + b0 + tb - 1, so the table id is uniform):
//   stage:  the tile's offsets go to shared memory; then every (id, chunk)
//           pair of the tile is hashed ONCE, by one thread, into a shared
//           array of block buckets x (loc = G*x).  Long tiles are staged in
//           chunks of `qc` ids.
//   gather / scatter: groups of gs lanes own consecutive bags of the tile and
//           walk their ids in order, U ids at a time so that U independent
//           16-byte loads per lane are in flight; a bag's row is stored when
//           its last id has been added (empty bags store zeros).
// Everything is index arithmetic on the CSR batch; no sort, no atomics in the
// forward.  The backward adds each bag's upstream-gradient row into every
// block the bag read (the dense branch of Algorithm 1) with global reductions:
// 16-byte fp32 vector reductions, or one fp64 reduction per element with
// consecutive lanes on consecutive elements (8 sectors per instruction).
#include <climits>

#include "pss_device.cuh"
#include "pss_internal.h"

namespace pss {
namespace {

constexpr int kU = 4;            // ids in flight per group
// ids in flight per group in the multi-id forward (4 or 8; measured on GB300
// at the multi-hot shape: 8 took 0.398 ms per forward with spills and 0.381
// at 3 CTAs per SM, against 0.334 ms with 4)
constexpr int kUM = 4;
static_assert(kUM == 4 || kUM == 8, "the multi-id forward sums 4 or 8 values per round as a tree");
constexpr int kBagsPerGroup = 16;
constexpr int kUB = 4;           // bags in flight per group in the forward's one-id path

template <typename XT>
struct Invalid;
template <>
struct Invalid<uint32_t> {
    static constexpr uint32_t v = 0xffffffffu;
};
template <>
struct Invalid<uint64_t> {
    static constexpr uint64_t v = ~uint64_t(0);
};

struct TileGeom {
    int tb;               // bags per tile
    int qc;               // ids per staging chunk
    int tiles_per_table;  // ceil(B / tb)
};

// Stage the offsets of tile (t, b0) into s_off; returns false (and zeroes the
// tile's rows when `out` is given) if the offsets are malformed.
// s_flags bit 0: malformed offsets; bit 1: some bag holds more than one id.
__device__ __forceinline__ bool stage_offsets(const int64_t* __restrict__ off, int64_t s0, int nb,
                                              int64_t nnz, int64_t* s_off, int* s_flags,
                                              DevError* err, bool* one_hot = nullptr) {
    if (threadIdx.x == 0) *s_flags = 0;
    for (int i = threadIdx.x; i <= nb; i += kThreads) s_off[i] = __ldg(off + s0 + i);
    __syncthreads();
    int f = 0;
    for (int i = threadIdx.x; i < nb; i += kThreads) {
        const int64_t a = s_off[i], c = s_off[i + 1];
        if (a < 0 || c < a || c > nnz) f |= 1;
        if (c - a > 1) f |= 2;
    }
    if (f) atomicOr(s_flags, f);
    __syncthreads();
    const int flags = *s_flags;
    if ((flags & 1) && threadIdx.x == 0) record_bad_offsets(err);
    if (one_hot) *one_hot = (flags & 2) == 0;
    return !(flags & 1);
}

// Hash every (id, chunk) pair of ids [qc0, qc0 + nq) of table t into s_x
// (CTA-cooperative; used by the atomic backward scatter).  With TOUCH every
// distinct bucket is also recorded in the touched bitmap / list, with one
// list-counter atomic per warp.
template <typename XT, bool TOUCH>
__device__ __forceinline__ void stage_buckets(const DevParams& p, const int64_t* __restrict__ idx,
                                              int t, uint64_t card, int64_t qc0, int nq, XT* s_x,
                                              DevError* err, const Touched& tc) {
    const int npairs = nq * p.J;
    const int lane = threadIdx.x & 31;
    for (int base = threadIdx.x & ~31; base < npairs; base += kThreads) {   // warp-uniform
        const int k = base + lane;
        XT x = Invalid<XT>::v;
        if (k < npairs) {
            const int qi = k / p.J;
            const int j = k - qi * p.J;
            const int64_t q = qc0 + qi;
            const int64_t id = __ldg(idx + q);
            if ((uint64_t)id < card) {
                const uint64_t key = hash_key(p, (uint64_t)id, t, j);
                x = (XT)hash_bucket(p, key) | (XT)hash_sign_bit(p, key);
            } else if (j == 0) {
                record_bad_id(err, q);
            }
            s_x[k] = x;
        }
        if (TOUCH)
            mark_touched_warp(tc, (uint64_t)(x & ~(XT)p.smask), x != Invalid<XT>::v, lane);
    }
}

// One VW-wide load of a staged block (bucket x, column offset z); with signed
// hashing (SG) the bucket carries the sign in bit 31, applied to the value.
// G < 2^31 (an int32 of the API): with 32-bit buckets the element index is
// one 32 x 32 -> 64-bit multiply.
template <bool SG, typename V, typename XT>
__device__ __forceinline__ typename V::T gather(const float* __restrict__ w, uint64_t G, XT x, int z) {
    const XT xb = SG ? (x & ~(XT)0x80000000u) : x;
    const uint64_t e = (sizeof(XT) == 4) ? (uint64_t)(uint32_t)G * (uint32_t)xb + (uint32_t)z
                                         : G * (uint64_t)xb + (uint64_t)z;
    if (!SG) return V::ldg(w + e);
    return sign_by(V::ldg(w + e), (uint32_t)x & 0x80000000u);
}

// ---------------------------------------------------------------------------
// Forward.  Each WARP owns a tile of `wb` consecutive bags of one table and
// stages it in its own slice of shared memory, so warps never wait for each
// other (no CTA-wide barrier): the lanes hash the tile's (id, chunk) pairs
// 32 at a time, then the lane groups gather and sum-pool their bags.
constexpr int kWarpPairs = 512;   // staged pairs per warp and round

// Hash the pairs [0, nq*J) of ids qc0.. into s_x (warp-cooperative); emits
// the buckets for the sorted backward when asked.
template <typename XT, bool SG>
__device__ __forceinline__ void warp_stage(const DevParams& p, const int64_t* __restrict__ idx,
                                           int t, uint64_t card, int64_t qc0, int nq, XT* s_x,
                                           DevError* err, uint32_t* __restrict__ pair_x,
                                           int lane) {
    const int npairs = nq * p.J;
    const bool jpow2 = (p.J & (p.J - 1)) == 0;
    const int log2J = 31 - __clz(p.J);
    for (int base = 0; base < npairs; base += 32) {
        const int k = base + lane;
        XT x = Invalid<XT>::v;
        if (k < npairs) {
            const int qi = jpow2 ? (k >> log2J) : k / p.J;
            const int j = k - qi * p.J;
            const int64_t q = qc0 + qi;
            const int64_t id = __ldg(idx + q);
            if ((uint64_t)id < card) {
                const uint64_t key = hash_key(p, (uint64_t)id, t, j);
                x = (XT)hash_bucket(p, key);
                if (SG) x |= (XT)hash_sign_bit(p, key);
            } else if (j == 0) {
                record_bad_id(err, q);
            }
            s_x[k] = x;
            if (pair_x) pair_x[qc0 * p.J + k] = (uint32_t)x;
        }
    }
    __syncwarp();
}

// One-id tiles: stage by BAG.  s_x[bb*J + j] is the bucket of chunk j of the
// id of bag bb (Invalid for an empty bag or a bad id), so the gather needs no
// offsets; the id's output row is written here too.
template <typename XT, bool SG>
__device__ __forceinline__ void warp_stage_bags(const DevParams& p, const int64_t* __restrict__ idx,
                                                int t, uint64_t card, const int64_t* s_off, int nb,
                                                XT* s_x, DevError* err,
                                                uint32_t* __restrict__ pair_x,
                                                uint32_t* __restrict__ q_row, uint32_t row0,
                                                int lane) {
    const int npairs = nb * p.J;
    const bool jpow2 = (p.J & (p.J - 1)) == 0;
    const int log2J = 31 - __clz(p.J);
    for (int base = 0; base < npairs; base += 32) {
        const int k = base + lane;
        XT x = Invalid<XT>::v;
        if (k < npairs) {
            const int bb = jpow2 ? (k >> log2J) : k / p.J;
            const int j = k - bb * p.J;
            const int64_t q = s_off[bb];
            if (s_off[bb + 1] > q) {
                const int64_t id = __ldg(idx + q);
                if ((uint64_t)id < card) {
                    const uint64_t key = hash_key(p, (uint64_t)id, t, j);
                    x = (XT)hash_bucket(p, key);
                if (SG) x |= (XT)hash_sign_bit(p, key);
                } else if (j == 0) {
                    record_bad_id(err, q);
                }
                if (pair_x) pair_x[q * p.J + j] = (uint32_t)x;
                if (q_row && j == 0) q_row[q] = row0 + (uint32_t)bb * (uint32_t)p.T;
            }
            s_x[k] = x;
        }
    }
    __syncwarp();
}

template <int VW, int KC, typename XT, bool SG>
__global__ void __launch_bounds__(kThreads, (KC == 1) ? 4 : 1)
k_forward_warp(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
               const int64_t* __restrict__ off, int64_t B, const float* __restrict__ w,
               float* __restrict__ out, DevError* err, uint32_t* __restrict__ pair_x,
               uint32_t* __restrict__ q_row, int log2gs, int wb,
               int tiles_per_table, int64_t b_lo, int64_t b_hi) {
    pdl_prologue();
    using V = Vec<VW>;
    using VT = typename V::T;
    extern __shared__ __align__(16) unsigned char smem[];
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    int64_t* s_off = reinterpret_cast<int64_t*>(smem) + warp * (wb + 1);
    XT* s_x = reinterpret_cast<XT*>(reinterpret_cast<int64_t*>(smem) + kWarps * (wb + 1)) +
              warp * kWarpPairs;
    const int gs = 1 << log2gs;
    const int lg = lane & (gs - 1);
    const int g = lane >> log2gs;
    const int bpg = wb >> (5 - log2gs);      // bags per group
    const Cols<VW, KC> col(p, lg, gs);
    const uint64_t G = (uint64_t)p.G;
    const int J = p.J;
    const int qcw = kWarpPairs / J;          // ids per staging round
    const int64_t ntiles = (int64_t)p.T * tiles_per_table;
    const int64_t ostride = (int64_t)p.T * p.d;

    for (int64_t tile = (int64_t)blockIdx.x * kWarps + warp; tile < ntiles;
         tile += (int64_t)gridDim.x * kWarps) {
        // ntiles < 2^31 (checked by the launcher): 32-bit division
        const int t = (int)((uint32_t)tile / (uint32_t)tiles_per_table);
        const int64_t b0 = b_lo + (tile - (int64_t)t * tiles_per_table) * wb;
        const int nb = (int)((b_hi - b0) < wb ? (b_hi - b0) : wb);
        const int64_t s0 = (int64_t)t * B + b0;
        float* obase = out + ((b0 * p.T) + t) * (int64_t)p.d;
        const int gb0 = min(g * bpg, nb);
        const int gb1 = min(gb0 + bpg, nb);

        for (int i = lane; i <= nb; i += 32) s_off[i] = __ldg(off + s0 + i);
        __syncwarp();
        bool bad = false, multi = false;
        for (int i = lane; i < nb; i += 32) {
            const int64_t a = s_off[i], c = s_off[i + 1];
            bad |= (a < 0 || c < a || c > nnz);
            multi |= (c - a > 1);
        }
        bad = __any_sync(0xffffffffu, bad);
        multi = __any_sync(0xffffffffu, multi);
        if (bad) {
            if (lane == 0) record_bad_offsets(err);
            for (int bi = gb0; bi < gb1; ++bi)
#pragma unroll
                for (int k = 0; k < KC; ++k) {
                    if (!col.v[k]) continue;
                    VT z;
#pragma unroll
                    for (int i = 0; i < VW; ++i) V::set(z, i, 0.f);
                    V::stcs(obase + bi * ostride + col.e[k], z);
                }
            __syncwarp();
            continue;
        }
        const uint64_t card = (uint64_t)__ldg(p.cards + t);
        const int64_t qb = s_off[nb];

        if (!multi && nb * J <= kWarpPairs) {
            // every bag holds at most one id: one load per bag, no accumulation
            warp_stage_bags<XT, SG>(p, idx, t, card, s_off, nb, s_x, err, pair_x, q_row,
                                (uint32_t)(b0 * p.T + t), lane);
            float* orow0 = obase + gb0 * ostride;
            for (int bb0 = gb0; bb0 < gb1; bb0 += kUB) {
                VT v[kUB][KC];
#pragma unroll
                for (int u = 0; u < kUB; ++u) {
                    const int bb = bb0 + u;
#pragma unroll
                    for (int k = 0; k < KC; ++k) {
#pragma unroll
                        for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                        if (bb < gb1 && col.v[k]) {
                            const XT x = s_x[bb * J + col.j[k]];
                            if (x != Invalid<XT>::v) v[u][k] = gather<SG, V>(w, G, x, col.z[k]);
                        }
                    }
                }
#pragma unroll
                for (int u = 0; u < kUB; ++u) {
                    if (bb0 + u >= gb1) break;
#pragma unroll
                    for (int k = 0; k < KC; ++k)
                        if (col.v[k]) V::stcs(orow0 + col.e[k], v[u][k]);
                    orow0 += ostride;
                }
            }
            __syncwarp();
            continue;
        }

        // general bags: the whole warp takes one bag at a time; its ng lane
        // groups add ng consecutive ids of the bag in parallel, kUM steps per
        // round.  A round's kUM values are summed as a tree and added to the
        // running sum with compensation (Kahan); at the end of the bag the
        // groups' sums are merged the same way and group 0 stores the row.
        const int ng = 32 >> log2gs;
        int64_t sw0 = 0, sw1 = 0;        // ids staged in s_x: [sw0, sw1)
        for (int bi = 0; bi < nb; ++bi) {
            const int64_t a = s_off[bi], c = s_off[bi + 1];
            float acc[KC][VW], cmp[KC][VW];
#pragma unroll
            for (int k = 0; k < KC; ++k)
#pragma unroll
                for (int i = 0; i < VW; ++i) acc[k][i] = cmp[k][i] = 0.f;
            const uint32_t row = (uint32_t)((b0 + bi) * p.T + t);
            for (int64_t q = a; q < c;) {
                if (q >= sw1) {
                    sw0 = q;
                    sw1 = (qb - q) < qcw ? qb : q + qcw;
                    warp_stage<XT, SG>(p, idx, t, card, sw0, (int)(sw1 - sw0), s_x, err, pair_x,
                                       lane);
                }
                const int64_t qend = c < sw1 ? c : sw1;
                // ids of the staged window by their 32-bit offset in it
                const int i1 = (int)(qend - sw0);
                for (int is = (int)(q - sw0); is < i1; is += kUM * ng) {
                    VT v[kUM][KC];
#pragma unroll
                    for (int u = 0; u < kUM; ++u) {
                        const int ii = is + u * ng + g;
#pragma unroll
                        for (int k = 0; k < KC; ++k) {
#pragma unroll
                            for (int i = 0; i < VW; ++i) V::set(v[u][k], i, 0.f);
                            if (ii < i1 && col.v[k]) {
                                const XT x = s_x[ii * J + col.j[k]];
                                if (x != Invalid<XT>::v) v[u][k] = gather<SG, V>(w, G, x, col.z[k]);
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < KC; ++k)
#pragma unroll
                        for (int i = 0; i < VW; ++i) {
                            float r = (V::get(v[0][k], i) + V::get(v[1][k], i)) +
                                      (V::get(v[2][k], i) + V::get(v[3][k], i));
                            if (kUM == 8)
                                r += (V::get(v[kUM / 2][k], i) + V::get(v[kUM / 2 + 1][k], i)) +
                                     (V::get(v[kUM - 2][k], i) + V::get(v[kUM - 1][k], i));
                            kahan_add(acc[k][i], cmp[k][i], r);
                        }
                }
                q = qend;
            }
            // the bag's ids' output row, one store per lane
            if (q_row)
                for (int64_t qq = a + lane; qq < c; qq += 32) q_row[qq] = row;
            for (int o = gs; o < 32; o <<= 1) {
#pragma unroll
                for (int k = 0; k < KC; ++k)
#pragma unroll
                    for (int i = 0; i < VW; ++i) {
                        const float os = __shfl_xor_sync(0xffffffffu, acc[k][i], o);
                        const float oc = __shfl_xor_sync(0xffffffffu, cmp[k][i], o);
                        kahan_add(acc[k][i], cmp[k][i], os);
                        kahan_add(acc[k][i], cmp[k][i], -oc);
                    }
            }
            if (g == 0) {
                float* orow = obase + bi * ostride;
#pragma unroll
                for (int k = 0; k < KC; ++k) {
                    if (!col.v[k]) continue;
                    VT o;
#pragma unroll
                    for (int i = 0; i < VW; ++i) V::set(o, i, acc[k][i] - cmp[k][i]);
                    V::stcs(orow + col.e[k], o);
                }
            }
        }
        __syncwarp();
    }
}

// ---------------------------------------------------------------------------
// Backward scatter: target[G*x + z] += scale * grad_out row chunk.
template <int VW, int KC, typename XT, typename AT, bool TOUCH>
__global__ void __launch_bounds__(kThreads)
k_scatter_tiled(DevParams p, const int64_t* __restrict__ idx, int64_t nnz,
                const int64_t* __restrict__ off, int64_t B, const float* __restrict__ gout,
                float scale, AT* __restrict__ target, Touched tc, DevError* err, int log2gs,
                TileGeom tg) {
    pdl_prologue();
    using V = Vec<VW>;
    using VT = typename V::T;
    extern __shared__ __align__(16) unsigned char smem[];
    int64_t* s_off = reinterpret_cast<int64_t*>(smem);
    XT* s_x = reinterpret_cast<XT*>(s_off + tg.tb + 1);
    __shared__ int s_bad;

    const int lane = threadIdx.x & 31;
    const int gs = 1 << log2gs;
    const int lg = lane & (gs - 1);
    const int grp = (threadIdx.x >> 5) * (32 >> log2gs) + (lane >> log2gs);
    const Cols<VW, KC> col(p, lg, gs);
    const uint64_t G = (uint64_t)p.G;
    const int J = p.J;
    const int64_t ntiles = (int64_t)p.T * tg.tiles_per_table;

    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int t = (int)(tile / tg.tiles_per_table);
        const int64_t b0 = (tile - (int64_t)t * tg.tiles_per_table) * tg.tb;
        const int nb = (int)((B - b0) < tg.tb ? (B - b0) : tg.tb);
        const int64_t s0 = (int64_t)t * B + b0;
        const int gb0 = min(grp * kBagsPerGroup, nb);
        const int gb1 = min(gb0 + kBagsPerGroup, nb);
        const float* gbase = gout + ((b0 * p.T) + t) * (int64_t)p.d;
        const int64_t gstride = (int64_t)p.T * p.d;

        if (!stage_offsets(off, s0, nb, nnz, s_off, &s_bad, err)) {
            __syncthreads();
            continue;
        }
        const uint64_t card = (uint64_t)__ldg(p.cards + t);
        const int64_t qa = s_off[0], qb = s_off[nb];
        const int64_t gq0 = s_off[gb0], gq1 = s_off[gb1];
        int bi = gb0;                       // bag of the next id
        int64_t qend = (gb0 < gb1) ? s_off[gb0 + 1] : 0;
        int have = -1;                      // bag whose row is in `row`
        VT row[KC];

        for (int64_t qc0 = qa; qc0 < qb; qc0 += tg.qc) {
            const int nq = (int)((qb - qc0) < tg.qc ? (qb - qc0) : tg.qc);
            stage_buckets<XT, TOUCH>(p, idx, t, card, qc0, nq, s_x, err, tc);
            __syncthreads();
            const int64_t qlo = gq0 > qc0 ? gq0 : qc0;
            const int64_t qhi = gq1 < qc0 + nq ? gq1 : qc0 + nq;
            for (int64_t q = qlo; q < qhi; q += kU) {
                // bags of the next kU ids, and their rows (independent loads)
                int ub[kU];
                VT r[kU][KC];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    ub[u] = -1;
                    if (q + u < qhi) {
                        while (q + u >= qend) {
                            ++bi;
                            qend = s_off[bi + 1];
                        }
                        ub[u] = bi;
                    }
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    if (ub[u] < 0) continue;
                    const bool same_prev = (u > 0) ? (ub[u] == ub[u - 1]) : (ub[u] == have);
                    if (same_prev) continue;
#pragma unroll
                    for (int k = 0; k < KC; ++k)
                        if (col.v[k])
                            r[u][k] = V::scale(V::ldcs(gbase + ub[u] * gstride + col.e[k]), scale);
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    if (ub[u] < 0) break;
                    const bool same_prev = (u > 0) ? (ub[u] == ub[u - 1]) : (ub[u] == have);
                    if (!same_prev) {
#pragma unroll
                        for (int k = 0; k < KC; ++k) row[k] = r[u][k];
                        have = ub[u];
                    }
#pragma unroll
                    for (int k = 0; k < KC; ++k) {
                        if (!col.v[k]) continue;
                        const XT x = s_x[(int)(q + u - qc0) * J + col.j[k]];
                        if (x != Invalid<XT>::v)
                            Acc<VW, AT>::red(target + G * (uint64_t)(x & ~(XT)p.smask) + col.z[k],
                                             sign_by(row[k], (uint32_t)x & p.smask));
                    }
                }
            }
            __syncthreads();
        }
        __syncthreads();
    }
}

TileGeom tile_geom(const DevParams& p, const RowLayout& lay, int64_t B, size_t xbytes) {
    TileGeom g;
    const int ng = 32 >> lay.log2gs;
    g.tb = kWarps * ng * kBagsPerGroup;
    const int stage_bytes = 16384;
    g.qc = stage_bytes / (int)(xbytes * (size_t)p.J);
    if (g.qc < 1) g.qc = 1;
    g.tiles_per_table = (int)((B + g.tb - 1) / g.tb);
    return g;
}

size_t tile_smem(const TileGeom& g, const DevParams& p, size_t xbytes) {
    return sizeof(int64_t) * (size_t)(g.tb + 1) + xbytes * (size_t)g.qc * (size_t)p.J;
}

template <int VW, int KC, typename XT, bool SG>
cudaError_t fwd_inst(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                     const int64_t* off, int64_t B, const float* w, float* out, DevError* err,
                     uint32_t* pair_x, uint32_t* q_row, int64_t b_lo, int64_t b_hi, int sm_count,
                     cudaStream_t st) {
    // bags per warp tile: kU per lane group (kU loads in flight in the one-id
    // path) and at least 16.  Measured on GB300: 16-bag tiles beat 32 and 64
    // at the Criteo-TB shape (0.165 against 0.171 and 0.174 ms per forward)
    // and on multi-id bags (0.385 against 0.419 ms), where the whole warp
    // takes one bag at a time; the 16-float rows of the Criteo-Kaggle shape
    // need the kU per group (batch 32768: 0.026 against 0.036 ms).
    const int groups = 32 >> lay.log2gs;
    const int wb = groups * kU > 16 ? groups * kU : 16;
    const int tpt = (int)((b_hi - b_lo + wb - 1) / wb);
    const size_t smem = (size_t)kWarps * ((size_t)(wb + 1) * sizeof(int64_t) +
                                          (size_t)kWarpPairs * sizeof(XT));
    const int64_t ntiles = (int64_t)p.T * tpt;
    if (ntiles >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;
    const int grid = grid_for(k_forward_warp<VW, KC, XT, SG>, sm_count, (ntiles + kWarps - 1) / kWarps,
                              smem);
    return launch_k(k_forward_warp<VW, KC, XT, SG>, dim3(grid), dim3(kThreads), smem, st, p, idx, nnz,
                    off, B, w, out, err, pair_x, q_row, lay.log2gs, wb, tpt, b_lo, b_hi);
}

template <int VW, int KC, typename XT, typename AT, bool TOUCH>
cudaError_t sc_inst(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                    const int64_t* off, int64_t B, const float* gout, float scale, AT* target,
                    const Touched& tc, DevError* err, int sm_count, cudaStream_t st) {
    const TileGeom tg = tile_geom(p, lay, B, sizeof(XT));
    const size_t smem = tile_smem(tg, p, sizeof(XT));
    const int64_t ntiles = (int64_t)p.T * tg.tiles_per_table;
    const int grid = grid_for(k_scatter_tiled<VW, KC, XT, AT, TOUCH>, sm_count, ntiles, smem);
    return launch_k(k_scatter_tiled<VW, KC, XT, AT, TOUCH>, dim3(grid), dim3(kThreads), smem, st, p,
                    idx, nnz, off, B, gout, scale, target, tc, err, lay.log2gs, tg);
}

template <int VW, int KC>
cudaError_t fwd_x(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                  const int64_t* off, int64_t B, const float* w, float* out, DevError* err,
                  uint32_t* pair_x, uint32_t* q_row, int64_t b_lo, int64_t b_hi, int sm_count,
                  cudaStream_t st) {
    if (p.R < 0xffffffffull)
        return p.smask ? fwd_inst<VW, KC, uint32_t, true>(p, lay, idx, nnz, off, B, w, out, err,
                                                           pair_x, q_row, b_lo, b_hi, sm_count, st)
                       : fwd_inst<VW, KC, uint32_t, false>(p, lay, idx, nnz, off, B, w, out, err,
                                                            pair_x, q_row, b_lo, b_hi, sm_count,
                                                            st);
    // R >= 2^32: 64-bit buckets, never signed (signed hashing needs R < 2^31)
    return fwd_inst<VW, KC, uint64_t, false>(p, lay, idx, nnz, off, B, w, out, err, nullptr,
                                             nullptr, b_lo, b_hi, sm_count, st);
}

template <int VW, int KC, typename AT>
cudaError_t sc_x(const DevParams& p, const RowLayout& lay, const int64_t* idx, int64_t nnz,
                 const int64_t* off, int64_t B, const float* gout, float scale, AT* target,
                 const Touched* tc, DevError* err, int sm_count, cudaStream_t st) {
    const Touched none{};
    const bool wide = p.R >= 0xffffffffull;
    if (tc) {
        if (wide)
            return sc_inst<VW, KC, uint64_t, AT, true>(p, lay, idx, nnz, off, B, gout, scale, target,
                                                        *tc, err, sm_count, st);
        return sc_inst<VW, KC, uint32_t, AT, true>(p, lay, idx, nnz, off, B, gout, scale, target,
                                                    *tc, err, sm_count, st);
    }
    if (wide)
        return sc_inst<VW, KC, uint64_t, AT, false>(p, lay, idx, nnz, off, B, gout, scale, target,
                                                     none, err, sm_count, st);
    return sc_inst<VW, KC, uint32_t, AT, false>(p, lay, idx, nnz, off, B, gout, scale, target, none,
                                                 err, sm_count, st);
}

}  // namespace

cudaError_t launch_forward(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* w, float* out,
                           DevError* err, uint32_t* pair_x, uint32_t* q_row, int64_t b_lo,
                           int64_t b_hi, int sm_count, cudaStream_t st) {
    if (b_lo < 0 || b_hi > B || b_lo >= b_hi) return cudaErrorInvalidValue;
#define PSS_FW(VW, KC)                                                                        \
    return fwd_x<VW, KC>(p, lay, idx, nnz, off, B, w, out, err, pair_x, q_row, b_lo, b_hi, \
                         sm_count, st)
    if (lay.vw == 4) {
        switch (lay.kc) {
            case 1: PSS_FW(4, 1);
            case 2: PSS_FW(4, 2);
            case 4: PSS_FW(4, 4);
        }
    } else {
        switch (lay.kc) {
            case 1: PSS_FW(1, 1);
            case 2: PSS_FW(1, 2);
            case 4: PSS_FW(1, 4);
            case 8: PSS_FW(1, 8);
            case 16: PSS_FW(1, 16);
        }
    }
#undef PSS_FW
    return cudaErrorInvalidValue;
}

cudaError_t launch_scatter(const DevParams& p, const RowLayout& lay, const int64_t* idx,
                           int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                           float scale, float* target, const Touched* touched, DevError* err,
                           int sm_count, cudaStream_t st) {
#define PSS_SC(VW, KC) \
    return sc_x<VW, KC, float>(p, lay, idx, nnz, off, B, grad_out, scale, target, touched, err, \
                               sm_count, st)
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

cudaError_t launch_scatter64(const DevParams& p, const RowLayout& lay_in, const int64_t* idx,
                             int64_t nnz, const int64_t* off, int64_t B, const float* grad_out,
                             double* target, const Touched* touched, DevError* err, int sm_count,
                             cudaStream_t st) {
    // fp64 reductions are scalar: lanes on consecutive elements
    const RowLayout lay = choose_layout(p.d, 1, 1);
    (void)lay_in;
#define PSS_SC(KC) \
    return sc_x<1, KC, double>(p, lay, idx, nnz, off, B, grad_out, 1.0f, target, touched, err, \
                               sm_count, st)
    switch (lay.kc) {
        case 1: PSS_SC(1);
        case 2: PSS_SC(2);
        case 4: PSS_SC(4);
        case 8: PSS_SC(8);
        case 16: PSS_SC(16);
    }
#undef PSS_SC
    return cudaErrorInvalidValue;
}

}  // namespace pss
