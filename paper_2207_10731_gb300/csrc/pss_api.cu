// C ABI of libpss.so (declared in include/pss.h): handle life cycle, argument
// validation, staging of host batches, backward-path dispatch and profiling.
#include <climits>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "pss.h"
#include "pss_internal.h"

using namespace pss;

namespace {

// Restores the caller's current device on scope exit.
struct DeviceGuard {
    int prev = -1;
    bool ok = false;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) == cudaSuccess) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

struct Staging {
    void* ptr = nullptr;
    size_t cap = 0;
};

struct EventPair {
    cudaEvent_t a, b;
};

}  // namespace

struct pss_handle {
    int device = 0;
    int sm_count = 0;
    int l2_bytes = 0;
    DevParams dp{};
    RowLayout layout{};
    std::vector<int64_t> cards;
    pss_optimizer opt = PSS_SGD;
    float eps = 1e-10f;

    float* w = nullptr;          // shared array M (library-owned)
    float* Gacc = nullptr;       // Adagrad accumulator
    float* g = nullptr;          // fp32 gradient accumulator, zero between calls
    double* g64 = nullptr;       // fp64 gradient accumulator, zero between calls
    int64_t* cards_dev = nullptr;
    DevError* err = nullptr;

    // batch of the last forward (device pointers: the caller's or staged)
    const int64_t* last_idx = nullptr;
    const int64_t* last_off = nullptr;
    int64_t last_nnz = 0, last_B = 0;
    bool have_batch = false;

    // options
    int64_t path = PSS_PATH_AUTO;
    int64_t update_mode = PSS_UPDATE_AUTO;
    int64_t profile = 0;
    int64_t sync_check = 0;
    int64_t accum = PSS_ACCUM_F64;
    int64_t sort_digit_bits = 0;                // PSS_OPT_SORT_DIGIT_BITS (0: automatic)
    int64_t deterministic = 0;                  // PSS_OPT_DETERMINISTIC
    int64_t sort_scope = PSS_SORT_AUTO;         // PSS_OPT_SORT_SCOPE
    int64_t last_path = PSS_PATH_ATOMIC;
    int64_t last_update = 0;                    // pss_info.last_update
    double last_collision = -1.0;

    Staging st_idx, st_off, st_out, st_grad, st_locs;

    // touched-block bookkeeping (allocated on first use)
    Touched touched{};
    int64_t touched_words = 0;

    // sorted backward path (allocated on first use)
    SortedBuffers sb{};
    int64_t sb_pairs_cap = 0, sb_ids_cap = 0;
    bool sb_fixed = false;                      // the buffers that do not grow with the batch
    bool sb_counting = false;                   // the counting sort's R-sized buffers
    int64_t radix_pairs_cap = 0;                // pairs the radix sort's buffers hold
    bool batch_emitted = false;                 // the last forward wrote pair_x / q_row
    unsigned long long* stats_host = nullptr;   // pinned mirror of sb.stats
    cudaEvent_t stats_ev = nullptr;
    // a host upstream gradient is copied in on s_h2d, which does not wait for
    // the caller's stream, so the copy overlaps the forward and the pooled
    // output's download; the caller's stream waits for ev_grad_ready just
    // before the first kernel that reads the gradient, and the next copy into
    // the staging buffer waits for ev_grad_free (its last reader)
    cudaStream_t s_h2d = nullptr;
    cudaEvent_t ev_grad_ready = nullptr, ev_grad_free = nullptr, ev_alloc = nullptr;
    bool grad_free_pending = false;
    // host-to-device copies of one direction run one after another on the
    // copy engine, so the gradient's upload also waits for the last forward's
    // staged ids and offsets (ev_inputs): otherwise those small copies queue
    // behind it and the forward and the output's download start only once
    // the whole gradient is in (measured: 9.1 ms per Criteo-TB step instead
    // of the 5.1 ms the two copy directions take together)
    cudaEvent_t ev_inputs = nullptr;
    bool inputs_pending = false;
    // a large pooled output bound for pinned host memory is computed in
    // chunks of batch rows, each downloaded on s_d2h as soon as its forward
    // kernel is done, so the download overlaps the following chunks' kernels;
    // the caller's stream then waits for the last download (ev_d2h)
    cudaStream_t s_d2h = nullptr;
    cudaEvent_t ev_fwd_chunk = nullptr, ev_d2h = nullptr;
    // circular array: R = M/G starts, blocks past M wrap to its start.  w and
    // the gradient accumulators have L extra elements past M: w's mirror
    // M[0 .. L) (refreshed after every write of w), the accumulators' collect
    // the wrapped contributions until they are folded into the head.
    bool circ = false;
    bool stats_pending = false;

    // profiling
    std::vector<EventPair> ev[PSS_K_COUNT];
    std::vector<EventPair> ev_free;
    int64_t launches_by_kernel[PSS_K_COUNT] = {0};
    int64_t launches = 0;
};

namespace {

pss_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return PSS_OK;
    if (e == cudaErrorMemoryAllocation) return PSS_ERR_OOM;
    return PSS_ERR_CUDA;
}

#define PSS_TRY(expr)                                  \
    do {                                               \
        pss_status _s = cuda_status(expr);             \
        if (_s != PSS_OK) return _s;                   \
    } while (0)

bool is_pinned_host_ptr(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeHost;
}

bool is_device_ptr(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

cudaError_t ensure(Staging& s, size_t bytes, cudaStream_t st) {
    if (bytes == 0) bytes = 16;
    if (s.cap >= bytes) return cudaSuccess;
    if (s.ptr) {
        cudaError_t e = cudaFreeAsync(s.ptr, st);
        if (e != cudaSuccess) return e;
        s.ptr = nullptr;
        s.cap = 0;
    }
    cudaError_t e = cudaMallocAsync(&s.ptr, bytes, st);
    if (e == cudaSuccess) s.cap = bytes;
    return e;
}

// Device view of a caller buffer: the pointer itself, or a staged copy.
template <typename T>
pss_status device_view(const T* p, size_t count, Staging& s, cudaStream_t st, const T** out) {
    if (count == 0 || is_device_ptr(p)) {
        *out = p;
        return PSS_OK;
    }
    PSS_TRY(ensure(s, count * sizeof(T), st));
    PSS_TRY(cudaMemcpyAsync(s.ptr, p, count * sizeof(T), cudaMemcpyHostToDevice, st));
    *out = static_cast<const T*>(s.ptr);
    return PSS_OK;
}

pss_status ensure_copy_stream(pss_handle* h) {
    if (h->s_h2d) return PSS_OK;
    PSS_TRY(cudaStreamCreateWithFlags(&h->s_h2d, cudaStreamNonBlocking));
    for (cudaEvent_t* e : {&h->ev_grad_ready, &h->ev_grad_free, &h->ev_alloc, &h->ev_inputs})
        PSS_TRY(cudaEventCreateWithFlags(e, cudaEventDisableTiming));
    return PSS_OK;
}

pss_status ensure_d2h_stream(pss_handle* h) {
    if (h->s_d2h) return PSS_OK;
    PSS_TRY(cudaStreamCreateWithFlags(&h->s_d2h, cudaStreamNonBlocking));
    for (cudaEvent_t* e : {&h->ev_fwd_chunk, &h->ev_d2h})
        PSS_TRY(cudaEventCreateWithFlags(e, cudaEventDisableTiming));
    return PSS_OK;
}

// Chunks of the forward when its output goes to pinned host memory: 4 from
// 64 MB of output on, else 1.  Measured end to end on GB300 over NVLink-C2C:
// Criteo-TB shape (872 MB of output) 0.299 -> 0.303 G lookups/s, multi-hot
// shape (109 MB, a longer forward) 4.67 -> 5.19 G lookups/s.
constexpr size_t kChunkedOutputBytes = size_t(64) << 20;
constexpr int kForwardChunks = 4;

// Device view of the upstream gradient.  A host buffer is copied into the
// staging buffer on s_h2d; *staged tells the caller to call grad_wait before
// the first kernel that reads it and grad_release after the last one.
pss_status stage_grad(pss_handle* h, const float* p, size_t count, cudaStream_t st,
                      const float** out, bool* staged) {
    *staged = false;
    if (count == 0 || is_device_ptr(p)) {
        *out = p;
        return PSS_OK;
    }
    pss_status rc = ensure_copy_stream(h);
    if (rc != PSS_OK) return rc;
    const size_t bytes = count * sizeof(float);
    if (h->st_grad.cap < bytes) {
        // (re)allocated in the caller's stream order; the copy waits for it
        PSS_TRY(ensure(h->st_grad, bytes, st));
        PSS_TRY(cudaEventRecord(h->ev_alloc, st));
        PSS_TRY(cudaStreamWaitEvent(h->s_h2d, h->ev_alloc, 0));
    }
    if (h->grad_free_pending) PSS_TRY(cudaStreamWaitEvent(h->s_h2d, h->ev_grad_free, 0));
    if (h->inputs_pending) {
        PSS_TRY(cudaStreamWaitEvent(h->s_h2d, h->ev_inputs, 0));
        h->inputs_pending = false;
    }
    PSS_TRY(cudaMemcpyAsync(h->st_grad.ptr, p, bytes, cudaMemcpyHostToDevice, h->s_h2d));
    PSS_TRY(cudaEventRecord(h->ev_grad_ready, h->s_h2d));
    *out = static_cast<const float*>(h->st_grad.ptr);
    *staged = true;
    return PSS_OK;
}

pss_status grad_wait(pss_handle* h, bool staged, cudaStream_t st) {
    if (staged) PSS_TRY(cudaStreamWaitEvent(st, h->ev_grad_ready, 0));
    return PSS_OK;
}

// After the last reader of a staged gradient.  The caller's stream also waits
// for the copy here (again, if a reader already did), so that no path returns
// with the caller's host buffer still being read.
pss_status grad_release(pss_handle* h, bool staged, cudaStream_t st) {
    if (staged) {
        PSS_TRY(cudaStreamWaitEvent(st, h->ev_grad_ready, 0));
        PSS_TRY(cudaEventRecord(h->ev_grad_free, st));
        h->grad_free_pending = true;
    }
    return PSS_OK;
}

EventPair take_events(pss_handle* h) {
    if (!h->ev_free.empty()) {
        EventPair e = h->ev_free.back();
        h->ev_free.pop_back();
        return e;
    }
    EventPair e{nullptr, nullptr};
    cudaEventCreate(&e.a);
    cudaEventCreate(&e.b);
    return e;
}

// Bracket n launches of one kernel kind: counts them and, when profiling,
// records events on their stream.
struct LaunchScope {
    pss_handle* h;
    int k;
    cudaStream_t st;
    int n;
    EventPair ev{nullptr, nullptr};
    LaunchScope(pss_handle* h_, int k_, cudaStream_t st_, int n_ = 1) : h(h_), k(k_), st(st_), n(n_) {
        if (h->profile) {
            ev = take_events(h);
            cudaEventRecord(ev.a, st);
        }
    }
    ~LaunchScope() {
        h->launches += n;
        h->launches_by_kernel[k] += n;
        if (h->profile && ev.a) {
            cudaEventRecord(ev.b, st);
            h->ev[k].push_back(ev);
        }
    }
};

pss_status check_error_word(pss_handle* h, cudaStream_t st, int64_t* first_bad) {
    DevError e;
    PSS_TRY(cudaMemcpyAsync(&e, h->err, sizeof(e), cudaMemcpyDeviceToHost, st));
    PSS_TRY(cudaStreamSynchronize(st));
    DevError clear{ULLONG_MAX, 0u, 0u};
    PSS_TRY(cudaMemcpyAsync(h->err, &clear, sizeof(clear), cudaMemcpyHostToDevice, st));
    PSS_TRY(cudaStreamSynchronize(st));
    int64_t fb = (e.first_bad == ULLONG_MAX) ? -1 : (int64_t)e.first_bad;
    if (fb < 0 && (e.flags & kErrOffsets)) fb = -2;
    if (first_bad) *first_bad = fb;
    return (fb != -1) ? PSS_ERR_INDEX_RANGE : PSS_OK;
}

pss_status ensure_grad(pss_handle* h, cudaStream_t st) {
    if (h->accum == PSS_ACCUM_F32) {
        if (h->g) return PSS_OK;
        PSS_TRY(cudaMalloc(&h->g, sizeof(float) * (size_t)(h->dp.M + h->dp.L)));
        PSS_TRY(cudaMemsetAsync(h->g, 0, sizeof(float) * (size_t)(h->dp.M + h->dp.L), st));
        return PSS_OK;
    }
    if (h->g64) return PSS_OK;
    PSS_TRY(cudaMalloc(&h->g64, sizeof(double) * (size_t)(h->dp.M + h->dp.L)));
    PSS_TRY(cudaMemsetAsync(h->g64, 0, sizeof(double) * (size_t)(h->dp.M + h->dp.L), st));
    return PSS_OK;
}

// Buffers sized by the number of block starts R, released when R changes (they
// are allocated again on first use).  The caller has synchronised the device.
void release_r_buffers(pss_handle* h) {
    for (void* b : {(void*)h->touched.bitmap, (void*)h->touched.list, (void*)h->touched.count,
                    (void*)h->sb.ccnt, (void*)h->sb.start, (void*)h->sb.bsum, (void*)h->sb.bnz})
        if (b) cudaFree(b);
    h->sb.ccnt = h->sb.start = h->sb.bsum = h->sb.bnz = nullptr;
    h->sb_counting = false;
    h->touched = Touched{};
    h->touched_words = 0;
}

// Circular array: refresh w's mirror of M[0 .. L) after a write of w.
pss_status mirror_head(pss_handle* h, cudaStream_t st) {
    if (h->circ)
        PSS_TRY(cudaMemcpyAsync(h->w + h->dp.M, h->w, sizeof(float) * (size_t)h->dp.L,
                                cudaMemcpyDeviceToDevice, st));
    return PSS_OK;
}

// Circular array: fold the accumulator's wrapped contributions into its head.
pss_status fold_tail(pss_handle* h, bool f64, cudaStream_t st) {
    if (h->circ) {
        LaunchScope ls(h, PSS_K_MISC, st);
        PSS_TRY(launch_fold_tail(f64 ? h->g64 : nullptr, f64 ? nullptr : h->g, (int64_t)h->dp.M,
                                 h->dp.L, st));
    }
    return PSS_OK;
}

pss_status ensure_touched(pss_handle* h, int64_t pairs, cudaStream_t st) {
    const int64_t R = (int64_t)h->dp.R;
    int64_t need = pairs < R ? pairs : R;
    if (need < 1) need = 1;
    if (!h->touched.bitmap) {
        const int64_t extra = (int64_t)h->dp.L / h->dp.G + 64;
        h->touched_words = (R + extra) / 32 + 2;
        PSS_TRY(cudaMalloc(&h->touched.bitmap, sizeof(uint32_t) * (size_t)h->touched_words));
        PSS_TRY(cudaMemsetAsync(h->touched.bitmap, 0, sizeof(uint32_t) * (size_t)h->touched_words, st));
        PSS_TRY(cudaMalloc(&h->touched.count, sizeof(unsigned long long)));
        PSS_TRY(cudaMemsetAsync(h->touched.count, 0, sizeof(unsigned long long), st));
    }
    if (h->touched.cap < need) {
        if (h->touched.list) PSS_TRY(cudaFreeAsync(h->touched.list, st));
        h->touched.list = nullptr;
        h->touched.cap = 0;
        PSS_TRY(cudaMallocAsync(&h->touched.list, sizeof(int64_t) * (size_t)need, st));
        h->touched.cap = need;
    }
    return PSS_OK;
}

bool use_touched(const pss_handle* h, int64_t pairs) {
    if (h->circ) return false;   // the ownership rule of the touched pass does not wrap
    if (h->update_mode == PSS_UPDATE_DENSE) return false;
    if (h->update_mode == PSS_UPDATE_TOUCHED) return true;
    // the dense pass touches every element of M once; the touched pass visits
    // at most pairs*L elements at random, and clears its bitmap in a kernel of
    // its own.  While M's working set (w, the Adagrad accumulator and the fp64
    // gradient: 16 bytes per element) fits in half the L2, the dense pass wins
    // (measured on GB300: Criteo-Kaggle shape 0.020 against 0.026 ms per step,
    // Criteo-TB batch 64 0.035 against 0.038); beyond, the touched pass wins
    // once M exceeds pairs*L (M = 2^25, batch 1024: 0.061 against 0.104 ms).
    if (16 * h->dp.M <= (int64_t)h->l2_bytes / 2) return false;
    return h->dp.M > pairs * (int64_t)h->dp.L;
}

// The sorted path holds bucket indices in 32 bits, 0xffffffff marking a bad
// id: it needs R < kSortedMaxR, the bound below which the forward emits 32-bit
// buckets at all.  AUTO takes the sorted path when the batch adds at least
// auto_sorted_min_adds(L) elements (pairs * L), the atomic path below: the
// atomic path's one kernel wins small batches, the sorted path's sort and
// reduce win large ones at every M from 2^18 to 2^33, Zipf or uniform ids.
// Measured on GB300 (ms per step, atomic against sorted):
//   L = 32, Criteo-TB shape:     3.4M adds 0.045 / 0.055, 6.8M adds 0.074 / 0.059
//   L = 16, Criteo-Kaggle shape: 6.8M adds 0.087 / 0.118, 13.6M adds 0.186 / 0.138
// (blocks shorter than a warp leave the sorted reduce's lanes partly idle, so
// its crossover lies higher).
constexpr int64_t kSortedMaxR = int64_t(0xffffffffLL);

int64_t auto_sorted_min_adds(int32_t L) { return L >= 32 ? 5000000 : 10000000; }

bool sorted_supported(const pss_handle* h, int64_t nnz, int64_t B) {
    const int64_t J = h->dp.J;
    // entries hold row*J + j in 32 bits (31 with signed hashing: the sign
    // travels in bit 31)
    const int64_t lim = h->dp.smask ? (int64_t)0x7fffffffLL : (int64_t)0xffffffffLL;
    return (int64_t)h->dp.R < kSortedMaxR && nnz * J < (int64_t)0xffffffffLL &&
           (int64_t)h->dp.T * B * J < lim;
}

// The sorted path's sort: the counting sort (one counter per bucket), unless
// the caller asked for run-to-run identical bits or R exceeds its counters.
bool use_radix(const pss_handle* h) {
    return h->deterministic || (int64_t)h->dp.R > kCountSortMaxR;
}

bool want_sorted(const pss_handle* h, int64_t npairs) {
    if (h->path == PSS_PATH_SORTED) return true;
    if (h->path == PSS_PATH_ATOMIC) return false;
    return npairs * (int64_t)h->dp.L >= auto_sorted_min_adds(h->dp.L);
}

pss_status ensure_sorted(pss_handle* h, int64_t nnz, cudaStream_t st) {
    const int64_t npairs = nnz * h->dp.J;
    if (!h->sb_fixed) {
        PSS_TRY(cudaMalloc(&h->sb.stats, 2 * sizeof(unsigned long long)));
        PSS_TRY(cudaMemsetAsync(h->sb.stats, 0, 2 * sizeof(unsigned long long), st));
        PSS_TRY(cudaMallocHost(&h->stats_host, 2 * sizeof(unsigned long long)));
        h->stats_host[0] = h->stats_host[1] = 0;
        PSS_TRY(cudaEventCreateWithFlags(&h->stats_ev, cudaEventDisableTiming));
        h->sb_fixed = true;
    }
    if (h->sb_pairs_cap < npairs) {
        for (void** b : {(void**)&h->sb.pair_x, (void**)&h->sb.sorted_e, (void**)&h->sb.bnd,
                         (void**)&h->sb.segn}) {
            if (*b) PSS_TRY(cudaFreeAsync(*b, st));
            *b = nullptr;
        }
        h->sb_pairs_cap = 0;
        const size_t n = (size_t)(npairs > 0 ? npairs : 1);
        PSS_TRY(cudaMallocAsync(&h->sb.pair_x, sizeof(uint32_t) * n, st));
        PSS_TRY(cudaMallocAsync(&h->sb.sorted_e, sizeof(unsigned long long) * n, st));
        PSS_TRY(cudaMallocAsync(&h->sb.bnd, sizeof(float) * 64 * (size_t)window_records((int64_t)n),
                                st));
        PSS_TRY(cudaMallocAsync(&h->sb.segn, sizeof(uint32_t) * (size_t)local_segments((int64_t)n),
                                st));
        h->sb_pairs_cap = npairs;
    }
    if (h->sb_ids_cap < nnz) {
        if (h->sb.q_row) PSS_TRY(cudaFreeAsync(h->sb.q_row, st));
        h->sb.q_row = nullptr;
        h->sb_ids_cap = 0;
        PSS_TRY(cudaMallocAsync(&h->sb.q_row, sizeof(uint32_t) * (size_t)(nnz > 0 ? nnz : 1), st));
        h->sb_ids_cap = nnz;
    }
    return PSS_OK;
}

// The counting sort's buffers: one counter and one start per bucket.
pss_status ensure_counting(pss_handle* h, cudaStream_t st) {
    if (h->sb_counting) return PSS_OK;
    const int64_t R = (int64_t)h->dp.R;
    const int64_t nblk = sorted_scan_blocks(R);
    PSS_TRY(cudaMalloc(&h->sb.ccnt, sizeof(uint32_t) * (size_t)R));
    PSS_TRY(cudaMemsetAsync(h->sb.ccnt, 0, sizeof(uint32_t) * (size_t)R, st));
    PSS_TRY(cudaMalloc(&h->sb.start, sizeof(uint32_t) * (size_t)(R + 1)));
    PSS_TRY(cudaMalloc(&h->sb.bsum, sizeof(uint32_t) * (size_t)nblk));
    PSS_TRY(cudaMalloc(&h->sb.bnz, sizeof(uint32_t) * (size_t)nblk));
    h->sb_counting = true;
    return PSS_OK;
}

// The radix sort's buffers for npairs pairs: the second entry buffer and the
// per-tile digit counts of the widest digit.
pss_status ensure_radix(pss_handle* h, int64_t npairs, cudaStream_t st) {
    if (!h->sb.tot) {
        const size_t nd = size_t(1) << kRadixMaxBits;
        PSS_TRY(cudaMalloc(&h->sb.tot, sizeof(uint32_t) * nd));
        PSS_TRY(cudaMalloc(&h->sb.dstart, sizeof(uint32_t) * nd));
        PSS_TRY(cudaMalloc(&h->sb.done, sizeof(uint32_t)));
        PSS_TRY(cudaMemsetAsync(h->sb.done, 0, sizeof(uint32_t), st));
    }
    if (h->radix_pairs_cap < npairs) {
        for (void** b : {(void**)&h->sb.tmp_e, (void**)&h->sb.cnt}) {
            if (*b) PSS_TRY(cudaFreeAsync(*b, st));
            *b = nullptr;
        }
        h->radix_pairs_cap = 0;
        const size_t n = (size_t)(npairs > 0 ? npairs : 1);
        PSS_TRY(cudaMallocAsync(&h->sb.tmp_e, sizeof(unsigned long long) * n, st));
        const size_t nc = (size_t)radix_tiles((int64_t)n) * (size_t)(1 << kRadixMaxBits);
        PSS_TRY(cudaMallocAsync(&h->sb.cnt, sizeof(uint32_t) * nc, st));
        h->radix_pairs_cap = npairs;
    }
    return PSS_OK;
}

// Collision rate of the last sorted pass, once its statistics have arrived.
void poll_stats(pss_handle* h) {
    if (h->stats_pending && cudaEventQuery(h->stats_ev) == cudaSuccess) {
        const double pairs = (double)h->stats_host[0];
        h->last_collision = pairs > 0 ? 1.0 - (double)h->stats_host[1] / pairs : 0.0;
        h->stats_pending = false;
    }
    cudaGetLastError();
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

RowLayout layout_for(const pss_handle* h, const void* rowbuf) {
    if (h->layout.vw == 4 && !aligned16(rowbuf)) return choose_layout(h->dp.d, 1, 1);
    return h->layout;
}

pss_status validate_batch(const pss_handle* h, const int64_t* idx, int64_t nnz,
                          const int64_t* off, int64_t B) {
    if (!off || B < 0 || nnz < 0 || (nnz > 0 && !idx)) return PSS_ERR_INVALID_ARG;
    if (B > (INT64_MAX / 2) / h->dp.T) return PSS_ERR_INVALID_ARG;
    return PSS_OK;
}

}  // namespace

extern "C" {

pss_status pss_check_convert(int32_t direction, const void* in, void* out, int64_t n,
                             pss_stream stream) {
    if ((direction != 0 && direction != 1) || n < 0) return PSS_ERR_INVALID_ARG;
    if (n == 0) return PSS_OK;
    if (!in || !out || !is_device_ptr(in) || !is_device_ptr(out)) return PSS_ERR_INVALID_ARG;
    int dev = 0, sms = 0;
    PSS_TRY(cudaGetDevice(&dev));
    PSS_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    PSS_TRY(launch_convert(direction, in, out, n, sms, reinterpret_cast<cudaStream_t>(stream)));
    return PSS_OK;
}

const char* pss_status_string(pss_status s) {
    switch (s) {
        case PSS_OK: return "ok";
        case PSS_ERR_INVALID_ARG: return "invalid argument";
        case PSS_ERR_OOM: return "device out of memory";
        case PSS_ERR_CUDA: return "CUDA runtime error";
        case PSS_ERR_STATE: return "invalid call order";
        case PSS_ERR_INDEX_RANGE: return "id outside its table, or malformed offsets";
        case PSS_ERR_TIMEOUT: return "device wait timed out";
        case PSS_ERR_UNSUPPORTED: return "unsupported";
        case PSS_ERR_CAPACITY:
            return "exceeds the fixed scratch capacity of pss_grad_noalloc (M <= 4194304, "
                   "tables <= 4096)";
    }
    return "unknown status";
}

pss_status pss_create(const int64_t* cards, int32_t T, int32_t dim, int64_t M, int32_t Z,
                      int32_t G, uint64_t seed, pss_optimizer opt, float adagrad_eps,
                      pss_stream stream, pss_handle** out) {
    if (!out || !cards || T <= 0 || dim <= 0 || dim > 512 || Z <= 0 || G <= 0 || M <= 0)
        return PSS_ERR_INVALID_ARG;
    if (opt != PSS_SGD && opt != PSS_ADAGRAD) return PSS_ERR_INVALID_ARG;
    if (opt == PSS_ADAGRAD && !(adagrad_eps > 0.f)) return PSS_ERR_INVALID_ARG;
    const int64_t J = (dim + Z - 1) / Z;
    const int64_t L = Z < dim ? Z : dim;
    if (M < L) return PSS_ERR_INVALID_ARG;
    int64_t max_card = 0;
    for (int32_t t = 0; t < T; ++t) {
        if (cards[t] <= 0) return PSS_ERR_INVALID_ARG;
        if (cards[t] > max_card) max_card = cards[t];
    }
    const unsigned __int128 P = (((unsigned __int128)1) << 61) - 1;
    if ((unsigned __int128)max_card * (unsigned __int128)T * (unsigned __int128)J > P)
        return PSS_ERR_INVALID_ARG;

    pss_handle* h = new (std::nothrow) pss_handle();
    if (!h) return PSS_ERR_OOM;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (cudaGetDevice(&h->device) != cudaSuccess) {
        delete h;
        return PSS_ERR_CUDA;
    }
    cudaDeviceGetAttribute(&h->sm_count, cudaDevAttrMultiProcessorCount, h->device);
    if (h->sm_count <= 0) h->sm_count = 1;
    cudaDeviceGetAttribute(&h->l2_bytes, cudaDevAttrL2CacheSize, h->device);

    DevParams& dp = h->dp;
    hash_params_from_seed(seed, &dp);
    dp.smask = 0u;
    dp.G = G;
    dp.M = M;
    dp.T = T;
    dp.d = dim;
    dp.Z = Z;
    dp.J = (int32_t)J;
    dp.L = (int32_t)L;
    dp.R = (uint64_t)((M - L) / G + 1);
    dp.Rinv = UINT64_MAX / dp.R;
    h->layout = choose_layout(dim, Z, G);
    h->cards.assign(cards, cards + T);
    h->opt = opt;
    h->eps = adagrad_eps;

    pss_status rc = PSS_OK;
    do {
        // L elements past M: the circular array's mirror of M[0 .. L)
        if ((rc = cuda_status(cudaMalloc(&h->w, sizeof(float) * (size_t)(M + L)))) != PSS_OK) break;
        if ((rc = cuda_status(cudaMemsetAsync(h->w, 0, sizeof(float) * (size_t)(M + L), st))) != PSS_OK)
            break;
        if (opt == PSS_ADAGRAD) {
            if ((rc = cuda_status(cudaMalloc(&h->Gacc, sizeof(float) * (size_t)M))) != PSS_OK) break;
            if ((rc = cuda_status(cudaMemsetAsync(h->Gacc, 0, sizeof(float) * (size_t)M, st))) != PSS_OK) break;
            if ((rc = ensure_grad(h, st)) != PSS_OK) break;
        }
        if ((rc = cuda_status(cudaMalloc(&h->cards_dev, sizeof(int64_t) * (size_t)T))) != PSS_OK) break;
        if ((rc = cuda_status(cudaMemcpy(h->cards_dev, cards, sizeof(int64_t) * (size_t)T,
                                         cudaMemcpyHostToDevice))) != PSS_OK) break;
        if ((rc = cuda_status(cudaMalloc(&h->err, sizeof(DevError)))) != PSS_OK) break;
        DevError clear{ULLONG_MAX, 0u, 0u};
        if ((rc = cuda_status(cudaMemcpy(h->err, &clear, sizeof(clear), cudaMemcpyHostToDevice))) != PSS_OK) break;
        if ((rc = cuda_status(cudaStreamSynchronize(st))) != PSS_OK) break;
    } while (0);
    dp.cards = h->cards_dev;
    if (rc != PSS_OK) {
        pss_destroy(h);
        return rc;
    }
    *out = h;
    return PSS_OK;
}

pss_status pss_destroy(pss_handle* h) {
    if (!h) return PSS_OK;
    DeviceGuard g(h->device);
    cudaDeviceSynchronize();
    cudaFree(h->w);
    cudaFree(h->Gacc);
    cudaFree(h->g);
    cudaFree(h->g64);
    cudaFree(h->cards_dev);
    cudaFree(h->err);
    cudaFree(h->touched.bitmap);
    cudaFree(h->touched.list);
    cudaFree(h->touched.count);
    for (void* b : {(void*)h->sb.pair_x, (void*)h->sb.q_row, (void*)h->sb.sorted_e,
                    (void*)h->sb.tmp_e, (void*)h->sb.cnt, (void*)h->sb.tot,
                    (void*)h->sb.dstart, (void*)h->sb.done, (void*)h->sb.stats,
                    (void*)h->sb.ccnt, (void*)h->sb.start, (void*)h->sb.bsum,
                    (void*)h->sb.bnz, (void*)h->sb.bnd, (void*)h->sb.segn})
        if (b) cudaFree(b);
    if (h->stats_host) cudaFreeHost(h->stats_host);
    if (h->stats_ev) cudaEventDestroy(h->stats_ev);
    for (cudaEvent_t e : {h->ev_grad_ready, h->ev_grad_free, h->ev_alloc, h->ev_inputs,
                          h->ev_fwd_chunk, h->ev_d2h})
        if (e) cudaEventDestroy(e);
    if (h->s_h2d) cudaStreamDestroy(h->s_h2d);
    if (h->s_d2h) cudaStreamDestroy(h->s_d2h);
    for (Staging* s : {&h->st_idx, &h->st_off, &h->st_out, &h->st_grad, &h->st_locs})
        if (s->ptr) cudaFree(s->ptr);
    for (int k = 0; k < PSS_K_COUNT; ++k)
        for (auto& e : h->ev[k]) {
            cudaEventDestroy(e.a);
            cudaEventDestroy(e.b);
        }
    for (auto& e : h->ev_free) {
        cudaEventDestroy(e.a);
        cudaEventDestroy(e.b);
    }
    delete h;
    return PSS_OK;
}

pss_status pss_set_weights(pss_handle* h, const float* w, int64_t n, pss_stream stream) {
    if (!h || !w || n != h->dp.M) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    PSS_TRY(cudaMemcpyAsync(h->w, w, sizeof(float) * (size_t)n, cudaMemcpyDefault,
                            reinterpret_cast<cudaStream_t>(stream)));
    return mirror_head(h, reinterpret_cast<cudaStream_t>(stream));
}

pss_status pss_get_weights(pss_handle* h, float* w, int64_t n, pss_stream stream) {
    if (!h || !w || n != h->dp.M) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    PSS_TRY(cudaMemcpyAsync(w, h->w, sizeof(float) * (size_t)n, cudaMemcpyDefault,
                            reinterpret_cast<cudaStream_t>(stream)));
    return PSS_OK;
}

pss_status pss_get_state(pss_handle* h, float* w, float* G, int64_t n, pss_stream stream) {
    if (!h || !w || n != h->dp.M || (h->opt == PSS_ADAGRAD && !G)) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    PSS_TRY(cudaMemcpyAsync(w, h->w, sizeof(float) * (size_t)n, cudaMemcpyDefault, st));
    if (h->opt == PSS_ADAGRAD)
        PSS_TRY(cudaMemcpyAsync(G, h->Gacc, sizeof(float) * (size_t)n, cudaMemcpyDefault, st));
    return PSS_OK;
}

pss_status pss_set_state(pss_handle* h, const float* w, const float* G, int64_t n,
                         pss_stream stream) {
    if (!h || !w || n != h->dp.M || (h->opt == PSS_ADAGRAD && !G)) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    PSS_TRY(cudaMemcpyAsync(h->w, w, sizeof(float) * (size_t)n, cudaMemcpyDefault, st));
    if (h->opt == PSS_ADAGRAD)
        PSS_TRY(cudaMemcpyAsync(h->Gacc, G, sizeof(float) * (size_t)n, cudaMemcpyDefault, st));
    return mirror_head(h, st);
}

pss_status pss_compute_locations(pss_handle* h, const int64_t* indices, int64_t nnz,
                                 const int64_t* offsets, int64_t B, int64_t* locs,
                                 pss_stream stream) {
    if (!h) return PSS_ERR_INVALID_ARG;
    pss_status rc = validate_batch(h, indices, nnz, offsets, B);
    if (rc != PSS_OK) return rc;
    if (nnz > 0 && !locs) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int64_t nbags = (int64_t)h->dp.T * B;
    const int64_t *di = nullptr, *doff = nullptr;
    if ((rc = device_view(indices, (size_t)nnz, h->st_idx, st, &di)) != PSS_OK) return rc;
    if ((rc = device_view(offsets, (size_t)(nbags + 1), h->st_off, st, &doff)) != PSS_OK) return rc;
    const size_t nloc = (size_t)nnz * (size_t)h->dp.J;
    int64_t* dl = locs;
    const bool host_out = nloc > 0 && !is_device_ptr(locs);
    if (host_out) {
        PSS_TRY(ensure(h->st_locs, nloc * sizeof(int64_t), st));
        dl = static_cast<int64_t*>(h->st_locs.ptr);
        PSS_TRY(cudaMemcpyAsync(dl, locs, nloc * sizeof(int64_t), cudaMemcpyHostToDevice, st));
    }
    if (nbags > 0) {
        LaunchScope ls(h, PSS_K_LOCATIONS, st);
        PSS_TRY(launch_locations(h->dp, di, nnz, doff, B, dl, h->err, h->sm_count, st));
    }
    if (host_out)
        PSS_TRY(cudaMemcpyAsync(locs, dl, nloc * sizeof(int64_t), cudaMemcpyDeviceToHost, st));
    if (h->sync_check) return check_error_word(h, st, nullptr);
    return PSS_OK;
}

pss_status pss_forward(pss_handle* h, const int64_t* indices, int64_t nnz, const int64_t* offsets,
                       int64_t B, float* out, pss_stream stream) {
    if (!h) return PSS_ERR_INVALID_ARG;
    pss_status rc = validate_batch(h, indices, nnz, offsets, B);
    if (rc != PSS_OK) return rc;
    const int64_t nbags = (int64_t)h->dp.T * B;
    if (nbags > 0 && !out) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int64_t *di = nullptr, *doff = nullptr;
    if ((rc = device_view(indices, (size_t)nnz, h->st_idx, st, &di)) != PSS_OK) return rc;
    if ((rc = device_view(offsets, (size_t)(nbags + 1), h->st_off, st, &doff)) != PSS_OK) return rc;
    if (di != indices || doff != offsets) {
        // host batch staged on st: a host gradient's upload waits for it
        if ((rc = ensure_copy_stream(h)) != PSS_OK) return rc;
        PSS_TRY(cudaEventRecord(h->ev_inputs, st));
        h->inputs_pending = true;
    }
    const size_t nout = (size_t)nbags * (size_t)h->dp.d;
    float* dout = out;
    const bool host_out = nout > 0 && !is_device_ptr(out);
    if (host_out) {
        PSS_TRY(ensure(h->st_out, nout * sizeof(float), st));
        dout = static_cast<float*>(h->st_out.ptr);
    }
    const bool emit =
        nbags > 0 && want_sorted(h, nnz * (int64_t)h->dp.J) && sorted_supported(h, nnz, B);
    if (emit && (rc = ensure_sorted(h, nnz, st)) != PSS_OK) return rc;
    const int chunks = (host_out && nout * sizeof(float) >= kChunkedOutputBytes &&
                        B >= kForwardChunks && is_pinned_host_ptr(out))
                           ? kForwardChunks
                           : 1;
    if (chunks > 1 && (rc = ensure_d2h_stream(h)) != PSS_OK) return rc;
    if (nbags > 0) {
        LaunchScope ls(h, PSS_K_FORWARD, st, chunks);
        const RowLayout lay = layout_for(h, dout);
        const size_t row = (size_t)h->dp.T * (size_t)h->dp.d;   // floats per batch row
        for (int c = 0; c < chunks; ++c) {
            const int64_t b_lo = B * c / chunks, b_hi = B * (c + 1) / chunks;
            PSS_TRY(launch_forward(h->dp, lay, di, nnz, doff, B, h->w, dout, h->err,
                                   emit ? h->sb.pair_x : nullptr, emit ? h->sb.q_row : nullptr,
                                   b_lo, b_hi, h->sm_count, st));
            if (chunks > 1) {
                PSS_TRY(cudaEventRecord(h->ev_fwd_chunk, st));
                PSS_TRY(cudaStreamWaitEvent(h->s_d2h, h->ev_fwd_chunk, 0));
                PSS_TRY(cudaMemcpyAsync(out + (size_t)b_lo * row, dout + (size_t)b_lo * row,
                                        (size_t)(b_hi - b_lo) * row * sizeof(float),
                                        cudaMemcpyDeviceToHost, h->s_d2h));
            }
        }
    }
    h->batch_emitted = emit;
    if (chunks > 1) {
        PSS_TRY(cudaEventRecord(h->ev_d2h, h->s_d2h));
        PSS_TRY(cudaStreamWaitEvent(st, h->ev_d2h, 0));
    } else if (host_out) {
        PSS_TRY(cudaMemcpyAsync(out, dout, nout * sizeof(float), cudaMemcpyDeviceToHost, st));
    }
    h->last_idx = di;
    h->last_off = doff;
    h->last_nnz = nnz;
    h->last_B = B;
    h->have_batch = true;
    if (h->sync_check) return check_error_word(h, st, nullptr);
    return PSS_OK;
}

static pss_status scatter_into64(pss_handle* h, const float* dgrad, bool touch, cudaStream_t st) {
    const int64_t nbags = (int64_t)h->dp.T * h->last_B;
    if (nbags == 0) return PSS_OK;
    LaunchScope ls(h, PSS_K_SCATTER, st);
    return cuda_status(launch_scatter64(h->dp, layout_for(h, dgrad), h->last_idx, h->last_nnz,
                                        h->last_off, h->last_B, dgrad, h->g64,
                                        touch ? &h->touched : nullptr, h->err, h->sm_count, st));
}

static pss_status scatter_into(pss_handle* h, const float* dgrad, float scale, float* target,
                               bool touch, cudaStream_t st) {
    const int64_t nbags = (int64_t)h->dp.T * h->last_B;
    if (nbags == 0) return PSS_OK;
    // 16-byte vector atomics need both the gradient rows and the target aligned
    RowLayout lay = layout_for(h, dgrad);
    if (lay.vw == 4 && !aligned16(target)) lay = choose_layout(h->dp.d, 1, 1);
    LaunchScope ls(h, PSS_K_SCATTER, st);
    return cuda_status(launch_scatter(h->dp, lay, h->last_idx, h->last_nnz,
                                      h->last_off, h->last_B, dgrad, scale, target,
                                      touch ? &h->touched : nullptr, h->err, h->sm_count, st));
}

// Sorted path, step 1: sort the last forward's pairs by bucket (counting or
// radix sort); with `touch`, also list the touched blocks.
static pss_status sort_pairs(pss_handle* h, bool touch, bool local, cudaStream_t st) {
    const int64_t npairs = h->last_nnz * (int64_t)h->dp.J;
    poll_stats(h);
    if (local) {
        // grouped within segments only: no global count of distinct buckets
        LaunchScope ls(h, PSS_K_SORT, st, touch ? 2 : 1);
        PSS_TRY(launch_sort_local(h->sb, npairs, h->dp.J, h->dp.smask, h->sm_count, st));
        if (touch)
            PSS_TRY(launch_mark_pairs(h->sb, npairs, h->dp.smask, h->touched, h->sm_count, st));
        h->last_collision = -1.0;
    } else if (use_radix(h)) {
        pss_status rc0 = ensure_radix(h, npairs, st);
        if (rc0 != PSS_OK) return rc0;
        const RadixPlan plan = radix_plan(h->dp.R, (int)h->sort_digit_bits);
        LaunchScope ls(h, PSS_K_SORT, st, 3 * plan.passes + (touch ? 1 : 0));
        PSS_TRY(launch_radix_sort(h->sb, npairs, h->dp.J, h->dp.smask, plan, st));
        if (touch)
            PSS_TRY(launch_mark_pairs(h->sb, npairs, h->dp.smask, h->touched, h->sm_count, st));
    } else {
        // ccnt is zero here: it is zeroed when allocated, and every sort's scan
        // returns the counters it has read to zero
        pss_status rc0 = ensure_counting(h, st);
        if (rc0 != PSS_OK) return rc0;
        LaunchScope ls(h, PSS_K_SORT, st, 4);
        PSS_TRY(launch_sorted_count(h->sb, npairs, h->dp.smask, h->sm_count, st));
        PSS_TRY(launch_sorted_scan(h->sb, (int64_t)h->dp.R, touch ? &h->touched : nullptr, st));
        PSS_TRY(launch_sorted_scatter(h->sb, npairs, h->dp.J, h->dp.smask, h->sm_count, st));
    }
    return PSS_OK;
}

// Valid pairs (the sort) and distinct buckets (the reduce), for
// pss_get_info's collision rate; one copy in flight at a time.
static pss_status copy_stats(pss_handle* h, cudaStream_t st) {
    if (!h->stats_pending) {
        PSS_TRY(cudaMemcpyAsync(h->stats_host, h->sb.stats, 2 * sizeof(unsigned long long),
                                cudaMemcpyDeviceToHost, st));
        PSS_TRY(cudaEventRecord(h->stats_ev, st));
        h->stats_pending = true;
    }
    return PSS_OK;
}

// Sorted path with the window reduce: sort (with `touch`, also list the
// touched blocks), then every element's gradient stored once into gexp
// (fp32, zero on entry).
static pss_status sorted_window(pss_handle* h, const float* dgrad, bool staged, bool touch,
                                float* gexp, cudaStream_t st) {
    const int64_t npairs = h->last_nnz * (int64_t)h->dp.J;
    if (h->dp.T * h->last_B == 0 || npairs == 0) return grad_wait(h, staged, st);
    pss_status rc = sort_pairs(h, touch, false, st);
    if (rc != PSS_OK) return rc;
    if ((rc = grad_wait(h, staged, st)) != PSS_OK) return rc;
    {
        LaunchScope ls(h, PSS_K_REDUCE, st, 2);
        const WindowSink ws{gexp, h->sb.bnd};
        PSS_TRY(launch_window_reduce(h->sb, npairs, dgrad, h->dp, ws, h->sm_count, st));
    }
    return copy_stats(h, st);
}

// The fp32 gradient buffer of the window reduce (zero between calls).
static pss_status ensure_g32(pss_handle* h, cudaStream_t st) {
    if (h->g) return PSS_OK;
    PSS_TRY(cudaMalloc(&h->g, sizeof(float) * (size_t)(h->dp.M + h->dp.L)));
    PSS_TRY(cudaMemsetAsync(h->g, 0, sizeof(float) * (size_t)(h->dp.M + h->dp.L), st));
    return PSS_OK;
}

// Segment-local or global sort (PSS_OPT_SORT_SCOPE).  The local sort saves
// the global sort's per-bucket counters and atomics but leaves one run per
// bucket and segment, each an fp64 reduction of a chunk into g: it pays
// where few pairs share a block start, and above 2^22 starts, where the
// global sort is the radix sort.  Measured on GB300 (ms per step, global
// against local): Criteo-TB shape at 1.4, 2.7, 4.1 and 11 pairs per start
// 0.098/0.090, 0.152/0.153, 0.207/0.215, 0.465/0.495; paper micro-benchmark
// shape (1.7) 0.110/0.105; M = 2^22 at 3.3 per start 0.275/0.274; M = 2^24
// (1.6) 0.635/0.629; M = 2^28 (radix) 1.31/1.20.
static bool use_local_sort(const pss_handle* h, int64_t npairs, const float* dgrad) {
    if (h->deterministic || h->sort_scope == PSS_SORT_GLOBAL || !local_sort_ok(h->dp, dgrad))
        return false;
    if (h->sort_scope == PSS_SORT_LOCAL) return true;
    return (int64_t)h->dp.R > kCountSortMaxR ||
           npairs <= (int64_t)PSS_SORT_LOCAL_MAX_PAIRS_PER_START * (int64_t)h->dp.R;
}

// Sorted path: sort by bucket (segment-local, counting or radix), segmented
// reduce into g64.
static pss_status sorted_into64(pss_handle* h, const float* dgrad, bool staged, bool touch,
                                cudaStream_t st) {
    const int64_t npairs = h->last_nnz * (int64_t)h->dp.J;
    if (h->dp.T * h->last_B == 0 || npairs == 0) return PSS_OK;
    const bool local = use_local_sort(h, npairs, dgrad);
    pss_status rc0 = sort_pairs(h, touch, local, st);
    if (rc0 != PSS_OK) return rc0;
    // the sort above needs only the forward's buckets: a host gradient's copy
    // has overlapped it, and is waited for here
    pss_status rc = grad_wait(h, staged, st);
    if (rc != PSS_OK) return rc;
    {
        LaunchScope ls(h, PSS_K_REDUCE, st);
        PSS_TRY(launch_sorted_reduce(h->sb, npairs, dgrad, h->dp, h->g64, local,
                                     !local && use_radix(h), h->sm_count, st));
    }
    return local ? PSS_OK : copy_stats(h, st);
}

pss_status pss_backward_update(pss_handle* h, const float* grad_out, float lr, pss_stream stream) {
    if (!h) return PSS_ERR_INVALID_ARG;
    if (!h->have_batch) return PSS_ERR_STATE;
    const int64_t nbags = (int64_t)h->dp.T * h->last_B;
    if (nbags > 0 && !grad_out) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const float* dg = nullptr;
    bool staged = false;
    pss_status rc = stage_grad(h, grad_out, (size_t)nbags * (size_t)h->dp.d, st, &dg, &staged);
    if (rc != PSS_OK) return rc;
    const int64_t pairs = h->last_nnz * (int64_t)h->dp.J;
    const bool ada = h->opt == PSS_ADAGRAD;
    const bool sorted = h->batch_emitted && want_sorted(h, h->last_nnz * (int64_t)h->dp.J);
    h->last_path = sorted ? PSS_PATH_SORTED : PSS_PATH_ATOMIC;
    if (sorted && h->deterministic && !h->circ && window_reduce_ok(h->dp, dg)) {
        // each element's gradient stored once into the fp32 buffer, then the
        // update pass (which returns the buffer to zero)
        if ((rc = ensure_g32(h, st)) != PSS_OK) return rc;
        const bool touch = use_touched(h, pairs);
        h->last_update = touch ? PSS_UPDATE_TOUCHED : PSS_UPDATE_DENSE;
        if (touch && (rc = ensure_touched(h, pairs, st)) != PSS_OK) return rc;
        if ((rc = sorted_window(h, dg, staged, touch, h->g, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
        {
            LaunchScope ls(h, PSS_K_UPDATE, st);
            if (touch)
                PSS_TRY(launch_update_touched(ada, h->w, h->Gacc, h->g, h->touched, h->dp.G,
                                              h->dp.L, lr, h->eps, h->sm_count, st));
            else
                PSS_TRY(launch_update_dense(ada, h->w, h->Gacc, h->g, h->dp.M, lr, h->eps,
                                            h->sm_count, st));
        }
        if (touch) {
            LaunchScope ls(h, PSS_K_MISC, st);
            PSS_TRY(launch_touched_clear(h->touched, h->sm_count, st));
        }
    } else if (sorted) {
        const int64_t saved = h->accum;
        h->accum = PSS_ACCUM_F64;                 // the sorted path sums into g64
        rc = ensure_grad(h, st);
        h->accum = saved;
        if (rc != PSS_OK) return rc;
        const bool touch = use_touched(h, pairs);
        h->last_update = touch ? PSS_UPDATE_TOUCHED : PSS_UPDATE_DENSE;
        if (touch && (rc = ensure_touched(h, pairs, st)) != PSS_OK) return rc;
        if ((rc = sorted_into64(h, dg, staged, touch, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
        if ((rc = fold_tail(h, true, st)) != PSS_OK) return rc;
        {
            LaunchScope ls(h, PSS_K_UPDATE, st);
            if (touch)
                PSS_TRY(launch_update_touched64(ada, h->w, h->Gacc, h->g64, h->touched, h->dp.G,
                                                h->dp.L, lr, h->eps, h->sm_count, st));
            else
                PSS_TRY(launch_update_dense64(ada, h->w, h->Gacc, h->g64, h->dp.M, lr, h->eps,
                                              h->sm_count, st));
        }
        if (touch) {
            LaunchScope ls(h, PSS_K_MISC, st);
            PSS_TRY(launch_touched_clear(h->touched, h->sm_count, st));
        }
    } else if (h->accum == PSS_ACCUM_F32 && !ada && !h->circ) {
        // SGD is linear in g: scatter -lr * grad_out straight into M.
        h->last_update = 0;
        if ((rc = grad_wait(h, staged, st)) != PSS_OK) return rc;
        if (lr != 0.f && (rc = scatter_into(h, dg, -lr, h->w, false, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
    } else {
        if ((rc = ensure_grad(h, st)) != PSS_OK) return rc;
        const bool touch = use_touched(h, pairs);
        h->last_update = touch ? PSS_UPDATE_TOUCHED : PSS_UPDATE_DENSE;
        if (touch && (rc = ensure_touched(h, pairs, st)) != PSS_OK) return rc;
        if ((rc = grad_wait(h, staged, st)) != PSS_OK) return rc;
        if (h->accum == PSS_ACCUM_F32)
            rc = scatter_into(h, dg, 1.0f, h->g, touch, st);
        else
            rc = scatter_into64(h, dg, touch, st);
        if (rc != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
        if ((rc = fold_tail(h, h->accum != PSS_ACCUM_F32, st)) != PSS_OK) return rc;
        {
            LaunchScope ls(h, PSS_K_UPDATE, st);
            if (h->accum == PSS_ACCUM_F32) {
                if (touch)
                    PSS_TRY(launch_update_touched(ada, h->w, h->Gacc, h->g, h->touched, h->dp.G,
                                                  h->dp.L, lr, h->eps, h->sm_count, st));
                else
                    PSS_TRY(launch_update_dense(ada, h->w, h->Gacc, h->g, h->dp.M, lr, h->eps,
                                                h->sm_count, st));
            } else {
                if (touch)
                    PSS_TRY(launch_update_touched64(ada, h->w, h->Gacc, h->g64, h->touched,
                                                    h->dp.G, h->dp.L, lr, h->eps, h->sm_count, st));
                else
                    PSS_TRY(launch_update_dense64(ada, h->w, h->Gacc, h->g64, h->dp.M, lr, h->eps,
                                                  h->sm_count, st));
            }
        }
        if (touch) {
            LaunchScope ls(h, PSS_K_MISC, st);
            PSS_TRY(launch_touched_clear(h->touched, h->sm_count, st));
        }
    }
    if ((rc = mirror_head(h, st)) != PSS_OK) return rc;
    if (h->sync_check) return check_error_word(h, st, nullptr);
    return PSS_OK;
}

pss_status pss_backward_grad(pss_handle* h, const float* grad_out, float* grad, pss_stream stream) {
    if (!h || !grad) return PSS_ERR_INVALID_ARG;
    if (!h->have_batch) return PSS_ERR_STATE;
    const int64_t nbags = (int64_t)h->dp.T * h->last_B;
    if (nbags > 0 && !grad_out) return PSS_ERR_INVALID_ARG;
    if (!is_device_ptr(grad)) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const float* dg = nullptr;
    bool staged = false;
    pss_status rc = stage_grad(h, grad_out, (size_t)nbags * (size_t)h->dp.d, st, &dg, &staged);
    if (rc != PSS_OK) return rc;
    const bool sorted = h->batch_emitted && want_sorted(h, h->last_nnz * (int64_t)h->dp.J);
    h->last_path = sorted ? PSS_PATH_SORTED : PSS_PATH_ATOMIC;
    if (sorted && h->deterministic && !h->circ && window_reduce_ok(h->dp, dg)) {
        PSS_TRY(cudaMemsetAsync(grad, 0, sizeof(float) * (size_t)h->dp.M, st));
        if ((rc = sorted_window(h, dg, staged, false, grad, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
    } else if (sorted) {
        const int64_t saved = h->accum;
        h->accum = PSS_ACCUM_F64;
        rc = ensure_grad(h, st);
        h->accum = saved;
        if (rc != PSS_OK) return rc;
        if ((rc = sorted_into64(h, dg, staged, false, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
        if ((rc = fold_tail(h, true, st)) != PSS_OK) return rc;
        LaunchScope ls(h, PSS_K_MISC, st);
        PSS_TRY(launch_grad_export(h->g64, grad, h->dp.M, h->sm_count, st));
    } else if (h->accum == PSS_ACCUM_F32 && !h->circ) {
        PSS_TRY(cudaMemsetAsync(grad, 0, sizeof(float) * (size_t)h->dp.M, st));
        if ((rc = grad_wait(h, staged, st)) != PSS_OK) return rc;
        if ((rc = scatter_into(h, dg, 1.0f, grad, false, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
    } else {
        // (the circular array always takes the fp64 accumulator here: the
        // caller's grad has no room for the wrapped tail)
        const int64_t saved = h->accum;
        h->accum = PSS_ACCUM_F64;
        rc = ensure_grad(h, st);
        h->accum = saved;
        if (rc != PSS_OK) return rc;
        if ((rc = grad_wait(h, staged, st)) != PSS_OK) return rc;
        if ((rc = scatter_into64(h, dg, false, st)) != PSS_OK) return rc;
        if ((rc = grad_release(h, staged, st)) != PSS_OK) return rc;
        if ((rc = fold_tail(h, true, st)) != PSS_OK) return rc;
        LaunchScope ls(h, PSS_K_MISC, st);
        PSS_TRY(launch_grad_export(h->g64, grad, h->dp.M, h->sm_count, st));
    }
    if (h->sync_check) return check_error_word(h, st, nullptr);
    return PSS_OK;
}

pss_status pss_set_option(pss_handle* h, int32_t key, int64_t value) {
    if (!h) return PSS_ERR_INVALID_ARG;
    switch (key) {
        case PSS_OPT_BACKWARD_PATH:
            if (value < PSS_PATH_AUTO || value > PSS_PATH_SORTED) return PSS_ERR_INVALID_ARG;
            h->path = value;
            return PSS_OK;
        case PSS_OPT_UPDATE_MODE:
            if (value < PSS_UPDATE_AUTO || value > PSS_UPDATE_TOUCHED) return PSS_ERR_INVALID_ARG;
            h->update_mode = value;
            return PSS_OK;
        case PSS_OPT_PROFILE:
            if (value != 0 && value != 1) return PSS_ERR_INVALID_ARG;
            h->profile = value;
            return PSS_OK;
        case PSS_OPT_SYNC_CHECK:
            if (value != 0 && value != 1) return PSS_ERR_INVALID_ARG;
            h->sync_check = value;
            return PSS_OK;
        case PSS_OPT_ACCUM:
            if (value != PSS_ACCUM_F64 && value != PSS_ACCUM_F32) return PSS_ERR_INVALID_ARG;
            h->accum = value;
            return PSS_OK;
        case PSS_OPT_CIRCULAR: {
            if (value != 0 && value != 1) return PSS_ERR_INVALID_ARG;
            const int64_t M = h->dp.M, G = h->dp.G, L = h->dp.L;
            if (value && M % G) return PSS_ERR_UNSUPPORTED;
            const uint64_t R = value ? (uint64_t)(M / G) : (uint64_t)((M - L) / G + 1);
            if (h->dp.smask && R >= (uint64_t(1) << 31)) return PSS_ERR_UNSUPPORTED;
            if ((value != 0) == h->circ) return PSS_OK;
            DeviceGuard g(h->device);
            PSS_TRY(cudaDeviceSynchronize());
            release_r_buffers(h);
            h->dp.R = R;
            h->dp.Rinv = UINT64_MAX / R;
            h->circ = value != 0;
            h->have_batch = false;
            if (h->circ)
                PSS_TRY(cudaMemcpy(h->w + M, h->w, sizeof(float) * (size_t)L, cudaMemcpyDeviceToDevice));
            return PSS_OK;
        }
        case PSS_OPT_SIGNED: {
            if (value != 0 && value != 1) return PSS_ERR_INVALID_ARG;
            // the sign travels in bit 31 of a 32-bit bucket index
            if (value && h->dp.R >= (uint64_t(1) << 31)) return PSS_ERR_UNSUPPORTED;
            const uint32_t m = value ? 0x80000000u : 0u;
            if (m != h->dp.smask) h->have_batch = false;
            h->dp.smask = m;
            return PSS_OK;
        }
        case PSS_OPT_SORT_DIGIT_BITS:
            if (value != 0 && (value < 4 || value > kRadixMaxBits)) return PSS_ERR_INVALID_ARG;
            h->sort_digit_bits = value;
            return PSS_OK;
        case PSS_OPT_DETERMINISTIC:
            if (value != 0 && value != 1) return PSS_ERR_INVALID_ARG;
            h->deterministic = value;
            return PSS_OK;
        case PSS_OPT_SORT_SCOPE:
            if (value != PSS_SORT_AUTO && value != PSS_SORT_GLOBAL && value != PSS_SORT_LOCAL)
                return PSS_ERR_INVALID_ARG;
            h->sort_scope = value;
            return PSS_OK;
    }
    return PSS_ERR_INVALID_ARG;
}

pss_status pss_get_option(pss_handle* h, int32_t key, int64_t* value) {
    if (!h || !value) return PSS_ERR_INVALID_ARG;
    switch (key) {
        case PSS_OPT_BACKWARD_PATH: *value = h->path; return PSS_OK;
        case PSS_OPT_UPDATE_MODE: *value = h->update_mode; return PSS_OK;
        case PSS_OPT_PROFILE: *value = h->profile; return PSS_OK;
        case PSS_OPT_SYNC_CHECK: *value = h->sync_check; return PSS_OK;
        case PSS_OPT_ACCUM: *value = h->accum; return PSS_OK;
        case PSS_OPT_SIGNED: *value = h->dp.smask ? 1 : 0; return PSS_OK;
        case PSS_OPT_CIRCULAR: *value = h->circ ? 1 : 0; return PSS_OK;
        case PSS_OPT_SORT_DIGIT_BITS: *value = h->sort_digit_bits; return PSS_OK;
        case PSS_OPT_DETERMINISTIC: *value = h->deterministic; return PSS_OK;
        case PSS_OPT_SORT_SCOPE: *value = h->sort_scope; return PSS_OK;
    }
    return PSS_ERR_INVALID_ARG;
}

pss_status pss_get_error(pss_handle* h, int64_t* first_bad_index, pss_stream stream) {
    if (!h) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    return check_error_word(h, reinterpret_cast<cudaStream_t>(stream), first_bad_index);
}

pss_status pss_get_info(pss_handle* h, pss_info* info) {
    if (!h || !info) return PSS_ERR_INVALID_ARG;
    poll_stats(h);
    info->T = h->dp.T;
    info->d = h->dp.d;
    info->M = h->dp.M;
    info->Z = h->dp.Z;
    info->G = h->dp.G;
    info->J = h->dp.J;
    info->L = h->dp.L;
    info->R = (int64_t)h->dp.R;
    info->A = h->dp.A;
    info->B0 = h->dp.B0;
    info->A2 = h->dp.A2;
    info->B2 = h->dp.B2;
    info->signed_hash = h->dp.smask ? 1 : 0;
    info->circular = h->circ ? 1 : 0;
    info->optimizer = h->opt;
    info->kernel_launches = h->launches;
    info->last_path = h->last_path;
    info->last_update = h->last_update;
    info->last_collision_rate = h->last_collision;
    return PSS_OK;
}

pss_status pss_get_profile(pss_handle* h, int32_t kernel, int64_t* launches, double* total_ms) {
    if (!h || kernel < 0 || kernel >= PSS_K_COUNT) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    double tot = 0.0;
    for (auto& e : h->ev[kernel]) {
        PSS_TRY(cudaEventSynchronize(e.b));
        float ms = 0.f;
        PSS_TRY(cudaEventElapsedTime(&ms, e.a, e.b));
        tot += ms;
    }
    if (launches) *launches = (int64_t)h->ev[kernel].size();
    if (total_ms) *total_ms = tot;
    return PSS_OK;
}

pss_status pss_reset_profile(pss_handle* h) {
    if (!h) return PSS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    for (int k = 0; k < PSS_K_COUNT; ++k) {
        for (auto& e : h->ev[k]) {
            cudaEventSynchronize(e.b);
            h->ev_free.push_back(e);
        }
        h->ev[k].clear();
    }
    return PSS_OK;
}

}  // extern "C"
