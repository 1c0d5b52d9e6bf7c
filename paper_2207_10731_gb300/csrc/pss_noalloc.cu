// pss_grad_noalloc: the gradient of the shared array for one batch, computed
// without allocating any device memory.
//
// Some callers cannot call cudaMalloc: code embedded in a host framework that
// owns the whole device-memory budget and forbids side allocations (a serving
// process that pre-partitions memory, a plugin running under another runtime's
// allocator), and latency-critical code that cannot accept the implicit device
// synchronisation an allocation may cause.  This entry point serves them: the
// caller passes every input and the output, and the fp64 accumulator the
// scatter needs lives in a file-scope device array of fixed size.
#include <climits>
#include <mutex>

#include "pss.h"
#include "pss_device.cuh"
#include "pss_internal.h"

using namespace pss;

namespace {

// Fixed capacities of the static scratch (held by every GPU that loads the
// library, until the process exits): 2^22 fp64 accumulators (32 MiB) and the
// cardinalities of up to 4096 tables.
constexpr int64_t kMaxM = int64_t(1) << 22;
constexpr int32_t kMaxTables = 4096;
constexpr int kMaxDevices = 64;

__device__ __align__(256) double g_accum[kMaxM];
__device__ __align__(256) int64_t g_cards[kMaxTables];
__device__ __align__(256) DevError g_err;

// Device addresses of the arrays above, looked up once per device.  In host
// code the names g_accum etc. are host-side stand-ins, never device addresses.
struct Symbols {
    bool ready = false;
    double* accum = nullptr;
    int64_t* cards = nullptr;
    DevError* err = nullptr;
};
Symbols g_symbols[kMaxDevices];
std::mutex g_symbols_mu;

pss_status symbols_for_current_device(Symbols* out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PSS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_symbols_mu);
    Symbols& s = g_symbols[dev];
    if (!s.ready) {
        Symbols t;
        if (cudaGetSymbolAddress(reinterpret_cast<void**>(&t.accum), g_accum) != cudaSuccess ||
            cudaGetSymbolAddress(reinterpret_cast<void**>(&t.cards), g_cards) != cudaSuccess ||
            cudaGetSymbolAddress(reinterpret_cast<void**>(&t.err), g_err) != cudaSuccess) {
            cudaGetLastError();
            return PSS_ERR_CUDA;
        }
        t.ready = true;
        s = t;
    }
    *out = s;
    return PSS_OK;
}

bool on_device(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// The table sizes reach the device as kernel arguments, kCardsPerLaunch per
// launch: no host-to-device copy (a copy from pageable host memory would make
// the calling thread wait for the work already queued on the stream).
constexpr int kCardsPerLaunch = 256;
struct CardsChunk {
    int64_t v[kCardsPerLaunch];
    int32_t first, n;
};

__global__ void k_load_cards(CardsChunk c, int64_t* __restrict__ dst) {
    pdl_prologue();
    for (int i = threadIdx.x; i < c.n; i += blockDim.x) dst[c.first + i] = c.v[i];
}

__global__ void k_error_report(const DevError* err, int64_t* first_bad) {
    pdl_prologue();
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        int64_t v = (err->first_bad == ULLONG_MAX) ? -1 : (int64_t)err->first_bad;
        if (v < 0 && (err->flags & kErrOffsets)) v = -2;
        *first_bad = v;
    }
}

}  // namespace

extern "C" pss_status pss_grad_noalloc(const int64_t* cards, int32_t T, int32_t dim, int64_t M,
                                       int32_t Z, int32_t G, uint64_t seed,
                                       const int64_t* indices, int64_t nnz,
                                       const int64_t* offsets, int64_t B, const float* grad_out,
                                       float* grad, int64_t* first_bad, pss_stream stream) {
    // host-side validation (no device work is queued on failure)
    if (!cards || T <= 0 || dim <= 0 || dim > 512 || Z <= 0 || G <= 0 || M <= 0 || B < 0 ||
        nnz < 0 || !offsets || !grad || (nnz > 0 && !indices))
        return PSS_ERR_INVALID_ARG;
    if (M > kMaxM || T > kMaxTables) return PSS_ERR_CAPACITY;
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
    if (B > (INT64_MAX / 2) / T) return PSS_ERR_INVALID_ARG;
    const int64_t nbags = (int64_t)T * B;
    // every batch buffer must already be device memory (nothing is staged)
    if (!on_device(offsets) || !on_device(grad) || (nnz > 0 && !on_device(indices)) ||
        (nbags > 0 && (!grad_out || !on_device(grad_out))) || (first_bad && !on_device(first_bad)))
        return PSS_ERR_INVALID_ARG;

    Symbols sym;
    pss_status rc = symbols_for_current_device(&sym);
    if (rc != PSS_OK) return rc;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);

    DevParams p{};
    hash_params_from_seed(seed, &p);
    p.G = G;
    p.M = M;
    p.T = T;
    p.d = dim;
    p.Z = Z;
    p.J = (int32_t)J;
    p.L = (int32_t)L;
    p.R = (uint64_t)((M - L) / G + 1);
    p.Rinv = UINT64_MAX / p.R;
    p.cards = sym.cards;

    // The scratch keeps the previous call's contents: clear what must start at
    // zero (the accumulator and the error word) and load the table sizes.
    if (cudaMemsetAsync(sym.accum, 0, sizeof(double) * (size_t)M, st) != cudaSuccess ||
        cudaMemsetAsync(&sym.err->first_bad, 0xff, sizeof(unsigned long long), st) != cudaSuccess ||
        cudaMemsetAsync(&sym.err->flags, 0, sizeof(unsigned int), st) != cudaSuccess)
        return PSS_ERR_CUDA;
    for (int32_t t0 = 0; t0 < T; t0 += kCardsPerLaunch) {
        CardsChunk c;
        c.first = t0;
        c.n = (T - t0) < kCardsPerLaunch ? (T - t0) : kCardsPerLaunch;
        for (int32_t i = 0; i < c.n; ++i) c.v[i] = cards[t0 + i];
        if (launch_k(k_load_cards, dim3(1), dim3(kCardsPerLaunch), 0, st, c, sym.cards) !=
            cudaSuccess)
            return PSS_ERR_CUDA;
    }

    int sms = 1;
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (nbags > 0) {
        RowLayout lay = choose_layout(dim, Z, G);
        if (lay.vw == 4 && (((uintptr_t)grad_out) & 15u)) lay = choose_layout(dim, 1, 1);
        if (launch_scatter64(p, lay, indices, nnz, offsets, B, grad_out, sym.accum, nullptr,
                             sym.err, sms, st) != cudaSuccess)
            return PSS_ERR_CUDA;
    }
    if (launch_grad_export(sym.accum, grad, M, sms, st) != cudaSuccess) return PSS_ERR_CUDA;
    if (first_bad) {
        if (launch_k(k_error_report, dim3(1), dim3(32), 0, st, sym.err, first_bad) != cudaSuccess)
            return PSS_ERR_CUDA;
    }
    return PSS_OK;
}
