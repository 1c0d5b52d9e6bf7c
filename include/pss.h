/*
 * pss.h -- C ABI of libpss.so: the hashed shared-array embedding ("parameter
 * sharing setup", PSS, with the ROBE-Z mapping) of Desai & Shrivastava, "The
 * trade-offs of model size in large recommendation models" (arXiv 2207.10731),
 * on one NVIDIA GB300 (sm_103a).
 *
 * The method (Def. 1, Sec. 2.1; Sec. 2.4; ROBE-Z mapping of Sec. 2.5):
 *   All T embedding tables share ONE learnable fp32 array M of length `M`.
 *   Chunk j (0 <= j < J, J = ceil(d/Z)) of the embedding of id i of table t is
 *   the contiguous block  M[loc(t,i,j) : loc(t,i,j) + L_j],  L_j = min(Z, d - jZ).
 *   A bag's output is the sum of the embeddings of its ids (sum pooling), so
 *       out[b][t][jZ + z] = sum over ids i of bag (t,b) of  M[loc(t,i,j) + z].
 *   The backward pass adds each bag's upstream gradient back into every block
 *   it read (the dense branch of Algorithm 1, Sec. 3), and the optimizer step
 *   (SGD or Adagrad) is applied to M in the same call.
 *
 * The location hash (Sec. 2.5 asks only for a universal hash; the choices below
 * are this library's, fixed so that results are reproducible bit for bit):
 *   P   = 2^61 - 1 (Mersenne prime)
 *   A   = 1 + (s1 mod (P-1)),  B0 = s2 mod P, where s1, s2 are the first two
 *         outputs of splitmix64 (Steele, Lea & Flood 2014) seeded with `seed`
 *   key = ((i*T + t)*J + j)                          (unsigned 64-bit)
 *   x   = (A*key + B0) mod P                         (exact, 128-bit product)
 *   L   = min(Z, d),   R = floor((M - L)/G) + 1
 *   loc = G * (x mod R)                              (so 0 <= loc <= M - L)
 *   G ("alignment") is the granularity of block starts: G = 4 makes every
 *   block 16-byte aligned; G = 1 is the paper's arbitrary offset.
 *
 * Batch layout (all int64, CSR, TABLE-MAJOR bags):
 *   bag (t, b) is slot s = t*B + b and owns indices[offsets[s] .. offsets[s+1]);
 *   offsets has T*B + 1 entries, non-decreasing, offsets[0] >= 0,
 *   offsets[T*B] <= nnz.  Pooled outputs and upstream gradients are fp32,
 *   row-major [B][T][d] (the DLRM concatenation order).
 *
 * Memory and streams:
 *   The library owns M, the Adagrad accumulator, its gradient scratch and all
 *   staging buffers; the caller owns every pointer it passes.  Calls taking a
 *   `stream` are asynchronous on it (stream-ordered) unless stated otherwise;
 *   the caller's buffers must stay valid until that work completes.  Batch
 *   pointers may be device memory or host memory (pinned or pageable): host
 *   batches are staged through library-owned device buffers.  Indices,
 *   offsets and the pooled output move on the call's stream; a host upstream
 *   gradient is copied on a stream of the library's own, so that the copy
 *   overlaps the forward and the output's download, and the call's stream
 *   waits for it before the first kernel that reads it.  Either way, once the
 *   call's stream has reached the end of the call's work, the library is done
 *   with the caller's buffers.  A handle is not thread-safe; use one handle
 *   per thread or lock.
 *
 * Errors: every call returns a pss_status; none aborts the process.  Bad
 * arguments are rejected on the host before any work is queued.  An id outside
 * [0, n_t) cannot be seen on the host; the device skips that id (it contributes
 * nothing) and records the smallest such position in a device error word,
 * which pss_get_error() reads and clears.
 */
#ifndef PSS_H_
#define PSS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pss_handle pss_handle;
/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* pss_stream;

typedef enum {
    PSS_OK = 0,
    PSS_ERR_INVALID_ARG = 1,   /* a size, pointer or option value is invalid */
    PSS_ERR_OOM = 2,           /* a device allocation failed */
    PSS_ERR_CUDA = 3,          /* a CUDA runtime call failed */
    PSS_ERR_STATE = 4,         /* call order violated (e.g. backward before forward) */
    PSS_ERR_INDEX_RANGE = 5,   /* the device saw an id outside its table, or bad offsets */
    PSS_ERR_TIMEOUT = 6,       /* a bounded device wait gave up */
    PSS_ERR_UNSUPPORTED = 7,   /* valid request this build does not implement */
    PSS_ERR_CAPACITY = 8       /* request exceeds a fixed capacity (pss_grad_noalloc) */
} pss_status;

typedef enum { PSS_SGD = 0, PSS_ADAGRAD = 1 } pss_optimizer;

/* Option keys for pss_set_option / pss_get_option. */
typedef enum {
    /* Backward path: the dense gradient of Algorithm 1 built with vector atomics
     * (PSS_PATH_ATOMIC), or the sorted path that reduces equal locations before
     * touching M (PSS_PATH_SORTED, Algorithm 1's sparse branch).  On the atomic
     * path the order of a location's contributions depends on the GPU's
     * scheduling, so low-order bits may differ between runs (within the
     * accumulation bound; dyadic inputs give identical bits).  The sorted path
     * groups the contributions by location and sums each location's run once
     * (see PSS_OPT_DETERMINISTIC for its order).  PSS_PATH_AUTO takes the
     * sorted path when the batch adds at least 5,000,000 elements (nnz * J *
     * L) with blocks of L >= 32 elements, 10,000,000 with shorter blocks, the
     * atomic one below (crossovers measured on GB300; M does not move them). */
    PSS_OPT_BACKWARD_PATH = 1,
    /* How the Adagrad step visits M: every element (PSS_UPDATE_DENSE), only the
     * blocks the batch touched (PSS_UPDATE_TOUCHED), or chosen from M and the
     * batch size (PSS_UPDATE_AUTO: dense while 16 * M bytes fit in half the
     * GPU's L2 or M <= nnz * J * L, touched otherwise).  Results are identical;
     * pss_info's last_update says which pass ran. */
    PSS_OPT_UPDATE_MODE = 2,
    /* 1: record CUDA events around every kernel (read with pss_get_profile). */
    PSS_OPT_PROFILE = 3,
    /* 1: forward/backward synchronise the stream and return
     * PSS_ERR_INDEX_RANGE at once when the device error word is set. */
    PSS_OPT_SYNC_CHECK = 4,
    /* Precision of the gradient accumulator of the atomic path.
     * PSS_ACCUM_F64 (default): every contribution is added in fp64 and the sum
     * is rounded to fp32 once, so the error does not grow with the number of
     * contributions (8 bytes of scratch per element of M).
     * PSS_ACCUM_F32: 16-byte fp32 vector reductions (4 bytes per element, and
     * SGD is scattered straight into M); the error of a recursive fp32 sum,
     * up to (n-1) * 2^-24 * sum|contributions| for an element with n of them. */
    PSS_OPT_ACCUM = 5,
    /* 1: signed hashing.  Every (table t, id i, chunk j) also gets a sign
     * s = +-1 from a second hash of the same family (Sec. 2.5 builds the sketch
     * from +-1 random projections; ROBE-Z itself has none):
     *   s = -1 when ((A2*key + B2) mod (2^61-1)) is odd, else +1,
     * key as for the location, A2 = 1 + (s3 mod (2^61-2)) and B2 = s4 mod
     * (2^61-1) from the third and fourth splitmix64 outputs of the seed.  The
     * forward adds s * block and the backward s * upstream gradient.
     * Needs R < 2^31 (PSS_ERR_UNSUPPORTED otherwise).  Changing it forgets the
     * last forward's batch (the next backward needs a new forward).
     * pss_compute_locations returns locations only; pss_grad_noalloc is
     * unsigned. */
    PSS_OPT_SIGNED = 6,
    /* 1: circular array, the other reading of the printed range of h
     * (Sec. 2.5): R = M / G block starts, and element z of the block at loc is
     * M[(loc + z) mod M], so blocks near the end wrap to the start of M.
     * Needs G to divide M (PSS_ERR_UNSUPPORTED otherwise).  The optimizer pass
     * is then always the dense one.  Changing it synchronises the device,
     * changes R (pss_get_info) and forgets the last forward's batch.
     * pss_grad_noalloc does not wrap. */
    PSS_OPT_CIRCULAR = 7,
    /* Digit width of the sorted path's radix sort (used with
     * PSS_OPT_DETERMINISTIC, and for a global sort above 2^22 block starts,
     * see PSS_OPT_SORT_SCOPE): 0 (default)
     * sorts the bucket indices (bit width of R - 1) in as few passes of at
     * most 11 bits as possible; 4 to 11 forces that many bits per pass (more
     * passes).  The sort is stable, so the result does not depend on it. */
    PSS_OPT_SORT_DIGIT_BITS = 8,
    /* 1: run-to-run identical bits on the sorted path.  The sorted path then
     * sorts with the stable radix sort (see PSS_OPT_SORT_DIGIT_BITS), which
     * orders the contributions of every location by pair; the reduce sums
     * them in that order; for 32-element chunks that tile the rows each
     * element's additions then follow a fixed order (no atomics), for other
     * shapes the few run sums of an element meet in fp64 (exact, hence in any
     * order, unless their magnitudes span more than about 2^26).  0 (default):
     * the faster counting or segment-local sort (PSS_OPT_SORT_SCOPE), whose
     * order within a location follows the GPU's scheduling (the sum is within
     * the same bound, but low-order bits may differ between runs).  The atomic
     * path is not affected. */
    PSS_OPT_DETERMINISTIC = 9,
    /* How the sorted path (when not deterministic) groups the pairs by
     * location.  PSS_SORT_GLOBAL: one sort of all pairs (counting sort up to
     * 2^22 block starts, radix sort above).  PSS_SORT_LOCAL: within segments
     * of 8192 consecutive pairs only, one run per location and segment (the
     * runs of a location meet in the fp64 accumulator); no per-location
     * state, any R; needs chunks that tile the rows (Z = 32, d a multiple of
     * 32, 16-byte aligned upstream gradient), else the global sort runs.
     * PSS_SORT_AUTO (default): local where it is served and either R > 2^22
     * or the batch has at most PSS_SORT_LOCAL_MAX_PAIRS_PER_START pairs per
     * block start (few repeats to merge across segments); global otherwise.
     * After a local pass pss_info's last_collision_rate is -1 (no distinct
     * locations are counted). */
    PSS_OPT_SORT_SCOPE = 10
} pss_option;



enum { PSS_ACCUM_F64 = 0, PSS_ACCUM_F32 = 1 };

enum { PSS_PATH_AUTO = 0, PSS_PATH_ATOMIC = 1, PSS_PATH_SORTED = 2 };
enum { PSS_UPDATE_AUTO = 0, PSS_UPDATE_DENSE = 1, PSS_UPDATE_TOUCHED = 2 };
enum { PSS_SORT_AUTO = 0, PSS_SORT_GLOBAL = 1, PSS_SORT_LOCAL = 2 };
#define PSS_SORT_LOCAL_MAX_PAIRS_PER_START 3

/* Kernel ids for pss_get_profile. */
typedef enum {
    PSS_K_LOCATIONS = 0,   /* hash only (pss_compute_locations) */
    PSS_K_FORWARD = 1,     /* fused hash + gather + sum-pool */
    PSS_K_SCATTER = 2,     /* backward: hash + vector-atomic scatter (+ fused SGD) */
    PSS_K_UPDATE = 3,      /* optimizer pass over M (dense or touched blocks) */
    PSS_K_SORT = 4,        /* sorted path: the counting sort's count, scan and slot
                              scatter, or the radix sort's passes (and, with the touched
                              update, the marking of the touched blocks) */
    PSS_K_REDUCE = 5,      /* sorted path: run sums into the fp64 accumulator */
    PSS_K_MISC = 6,        /* memsets and small helper kernels */
    PSS_K_COUNT = 7
} pss_kernel_id;

/* Read-only description of a handle. */
typedef struct {
    int64_t T, d, M, Z, G, J, L, R;
    uint64_t A, B0;            /* hash parameters derived from the seed */
    int64_t optimizer;         /* pss_optimizer */
    int64_t kernel_launches;   /* kernels this handle has launched so far */
    int64_t last_path;         /* PSS_PATH_ATOMIC / PSS_PATH_SORTED of the last backward */
    double last_collision_rate;/* 1 - distinct blocks / (nnz*J) of the last sorted pass
                                  whose counts have reached the host, or -1 */
    uint64_t A2, B2;           /* sign-hash parameters derived from the seed */
    int64_t signed_hash;       /* PSS_OPT_SIGNED */
    int64_t circular;          /* PSS_OPT_CIRCULAR */
    int64_t last_update;       /* optimizer pass of the last pss_backward_update:
                                  PSS_UPDATE_DENSE, PSS_UPDATE_TOUCHED, or 0 (none yet,
                                  or SGD with the fp32 accumulator, scattered into M) */
} pss_info;

/*
 * Create a PSS instance (Def. 1, Sec. 2.1; ROBE-Z mapping, Sec. 2.5).
 *   table_cardinalities: host, num_tables entries n_t >= 1 (ids of table t are
 *                        0 .. n_t - 1).  Copied; the caller keeps ownership.
 *   dim (d):  1 .. 512.   Z: chunk length >= 1.   G: block-start alignment >= 1.
 *   M:        shared-array length in fp32 elements, M >= min(Z, d); 64-bit.
 *   seed:     hash seed (see the header comment).
 *   opt:      PSS_SGD or PSS_ADAGRAD;  adagrad_eps: Adagrad epsilon (> 0).
 * M (and, for Adagrad, the accumulator) is allocated on the current device and
 * zero-filled on `stream`; load initial values with pss_set_weights.
 * Errors: PSS_ERR_INVALID_ARG (sizes, null pointers, max_t n_t * T * J > 2^61-1),
 * PSS_ERR_OOM, PSS_ERR_CUDA.  *out is set only on success.
 */
pss_status pss_create(const int64_t* table_cardinalities, int32_t num_tables, int32_t dim,
                      int64_t M, int32_t Z, int32_t G, uint64_t seed, pss_optimizer opt,
                      float adagrad_eps, pss_stream stream, pss_handle** out);

/* Free every device buffer of the handle (synchronises the device first). NULL is a no-op. */
pss_status pss_destroy(pss_handle* h);

/* Copy n == M fp32 values into the shared array.  `w` is host or device memory.
 * Errors: PSS_ERR_INVALID_ARG (NULL, n != M), PSS_ERR_CUDA. */
pss_status pss_set_weights(pss_handle* h, const float* w, int64_t n, pss_stream stream);

/* Copy the shared array out (n == M).  Stream-ordered: synchronise `stream`
 * before reading a host buffer. */
pss_status pss_get_weights(pss_handle* h, float* w, int64_t n, pss_stream stream);

/* Checkpoint: copy M and the Adagrad accumulator (n == M each) to / from the
 * caller.  `G` is ignored (may be NULL) for SGD.  Host or device pointers. */
pss_status pss_get_state(pss_handle* h, float* w, float* G, int64_t n, pss_stream stream);
pss_status pss_set_state(pss_handle* h, const float* w, const float* G, int64_t n,
                         pss_stream stream);

/*
 * The mapping matrix of Algorithm 1 ("locations from which the output was
 * accessed"): locs[q*J + j] = loc(t, indices[q], j) for every id position q of
 * every bag, as an element offset into M; -1 for an id outside [0, n_t)
 * (that position is also recorded in the error word).  Positions not covered
 * by any bag are left untouched.
 *   indices: int64[nnz], offsets: int64[T*B+1] (table-major), B >= 0,
 *   locs:    int64[nnz*J].  Device or host pointers.
 */
pss_status pss_compute_locations(pss_handle* h, const int64_t* indices, int64_t nnz,
                                 const int64_t* offsets, int64_t B, int64_t* locs,
                                 pss_stream stream);

/*
 * Forward pass (Sec. 2.4 forward(i) = (S e_i)^T M, sum-pooled per bag):
 *   out[b][t][k] = sum over q in bag (t,b) of M[loc(t, indices[q], k / Z) + k % Z].
 * An empty bag gives a zero row.  out: fp32[B*T*d], fully overwritten.
 * The batch (indices, offsets, nnz, B) is remembered by pointer for the next
 * pss_backward_update / pss_backward_grad: the caller must keep it unchanged
 * until that call's work has completed.  Host batches are staged (and `out`
 * copied back) on `stream`.
 */
pss_status pss_forward(pss_handle* h, const int64_t* indices, int64_t nnz,
                       const int64_t* offsets, int64_t B, float* out, pss_stream stream);

/*
 * Backward pass fused with the optimizer step for the batch of the last
 * pss_forward (Sec. 2.4 backward(i, D) = (S e_i) D; Algorithm 1; SGD / Adagrad):
 *   g[e] = sum over every (bag, id, chunk j, z) with loc + z == e of grad_out[b][t][jZ+z]
 *   SGD:     M[e] -= lr * g[e]
 *   Adagrad: G[e] += g[e]^2;  M[e] -= lr * g[e] / (sqrt(G[e]) + eps)   (only where g[e] != 0)
 * grad_out: fp32[B*T*d] (device or host).  lr: any finite value (lr = 0 leaves
 * M unchanged).  Errors: PSS_ERR_STATE if no forward has been run.
 */
pss_status pss_backward_update(pss_handle* h, const float* grad_out, float lr, pss_stream stream);

/*
 * Gradient only (Algorithm 1, dense branch output G_i): writes g (above) for
 * the batch of the last pss_forward into grad (fp32[M], DEVICE memory),
 * overwriting it; M and the optimizer state are not changed.
 */
pss_status pss_backward_grad(pss_handle* h, const float* grad_out, float* grad, pss_stream stream);

/* Set / get an option (pss_option).  Invalid key or value: PSS_ERR_INVALID_ARG. */
pss_status pss_set_option(pss_handle* h, int32_t key, int64_t value);
pss_status pss_get_option(pss_handle* h, int32_t key, int64_t* value);

/*
 * Synchronise `stream`, then read and clear the device error word.
 * *first_bad_index = smallest id position q seen outside its table since the
 * last call, or -1.  Returns PSS_ERR_INDEX_RANGE if an id or the offsets were
 * bad (offsets problems set *first_bad_index to -2 when no id was bad),
 * PSS_OK otherwise.
 */
pss_status pss_get_error(pss_handle* h, int64_t* first_bad_index, pss_stream stream);

/* Fill *info (host). */
pss_status pss_get_info(pss_handle* h, pss_info* info);

/*
 * Profiling (with PSS_OPT_PROFILE = 1): synchronise, then report for kernel id
 * `kernel` the number of launches and their summed device time in ms since the
 * last pss_reset_profile.  Times come from CUDA events recorded on the launch
 * stream immediately around each launch.
 */
pss_status pss_get_profile(pss_handle* h, int32_t kernel, int64_t* launches, double* total_ms);
pss_status pss_reset_profile(pss_handle* h);

/* Static description of a status code. */
const char* pss_status_string(pss_status s);

/*
 * Gradient of the shared array for one batch WITHOUT ALLOCATING device memory.
 * (The paper has no counterpart: this is a deployment aid of this library.)
 * For callers that cannot call cudaMalloc: code embedded in a host framework
 * that owns the whole device-memory budget and forbids side allocations, and
 * latency-critical code that cannot accept the implicit device synchronisation
 * an allocation may cause.  No handle is needed and nothing is allocated: the
 * caller passes every input and the output, and the fp64 accumulator lives in
 * a file-scope device array of fixed size, held by every GPU that loads the
 * library until the process exits.
 *   Computes, like pss_backward_grad with PSS_ACCUM_F64, for the mapping given
 *   by (table_cardinalities, num_tables, dim, M, Z, G, seed) as in pss_create:
 *     grad[e] = sum over every (bag, id, chunk j, z) with loc + z == e of grad_out[b][t][jZ+z]
 *   table_cardinalities: host, num_tables entries.  indices, offsets, grad_out,
 *   grad (fp32[M], overwritten) and first_bad: DEVICE memory (host pointers are
 *   rejected: nothing is staged).  first_bad (optional, int64[1]) receives the
 *   smallest position of an id outside its table (that id is skipped), -2 for
 *   malformed offsets, or -1.
 * Capacity: M <= 4194304 (2^22: 32 MiB of fp64 scratch) and num_tables <= 4096;
 * larger requests return PSS_ERR_CAPACITY before any device work is queued.
 * The first call on a device looks up the scratch's device address (once per
 * device, with that device current); make that first call before any stream
 * capture.  Every call shares the one scratch array: calls whose work overlaps
 * on the GPU (other streams, other threads) race and give wrong results, so
 * order them on one stream or synchronise between them.  Asynchronous on
 * `stream`: the call queues memsets of the scratch and a few kernels, and the
 * table sizes travel as kernel arguments, so nothing is copied from host
 * memory and the calling thread does not wait for work already on `stream`.
 * Errors: PSS_ERR_INVALID_ARG, PSS_ERR_CAPACITY, PSS_ERR_CUDA.
 */
pss_status pss_grad_noalloc(const int64_t* table_cardinalities, int32_t num_tables, int32_t dim,
                            int64_t M, int32_t Z, int32_t G, uint64_t seed,
                            const int64_t* indices, int64_t nnz, const int64_t* offsets,
                            int64_t B, const float* grad_out, float* grad, int64_t* first_bad,
                            pss_stream stream);

/*
 * Check of the two conversions of the fp64 gradient accumulation (the paper
 * has no counterpart: a test hook of this library).  direction 0: out[i] =
 * the fp32 value in[i] widened exactly to fp64 (in: float[n], out: double[n]);
 * direction 1: out[i] = fp64 in[i] rounded to the nearest fp32, ties to even
 * (in: double[n], out: float[n]).  Both are the integer-arithmetic routines the
 * kernels use, so a caller can compare them bit for bit with IEEE-754
 * conversions.  `in` and `out` are device buffers owned by the caller.
 * Asynchronous on `stream`.  Errors: PSS_ERR_INVALID_ARG (direction not 0 or
 * 1, n < 0, a null or host buffer), PSS_ERR_CUDA.
 */
pss_status pss_check_convert(int32_t direction, const void* in, void* out, int64_t n,
                             pss_stream stream);

/*
 * L2 rate probe (the paper has no counterpart: a measurement hook of this
 * library, used for the L2 roofline).  Queues one kernel of `ctas` CTAs of 256
 * threads on `stream` over the caller's DEVICE buffer `buf` of `bytes` bytes
 * (256-byte aligned, at least 4096; its contents are overwritten):
 *   kind 0: every warp reads `iters` (rounded up to a multiple of 8) random
 *           128-byte blocks of buf (lane l reads word l of the block), among
 *           the first power-of-two number of blocks that fits;
 *   kind 1: every warp adds 1.0 into `iters` random blocks of 32 consecutive
 *           doubles of buf, one per lane (red.global.add.f64), among the
 *           first power-of-two number of blocks that fits;
 *   kind 2: likewise (1,1,1,1) into blocks of 32 consecutive 16-byte fp32
 *           vectors (red.global.add.v4.f32);
 *   kind 3: like kind 0, but the warps read consecutive 128-byte lines
 *           (a streaming read of buf, wrapping around).
 * The caller times the call with events on `stream`; bytes moved = ctas * 8 *
 * iters * 128 (kinds 0 and 3), adds = ctas * 256 * iters (kind 1) or 4x that
 * (kind 2).  Buffers below 512 bytes per block are refused for kinds 1 and 2
 * only through the 4096-byte minimum.
 * Errors: PSS_ERR_INVALID_ARG (kind, sizes, alignment, a host buffer),
 * PSS_ERR_CUDA.
 */
pss_status pss_probe_l2(int32_t kind, void* buf, int64_t bytes, int64_t iters, int32_t ctas,
                        pss_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* PSS_H_ */
