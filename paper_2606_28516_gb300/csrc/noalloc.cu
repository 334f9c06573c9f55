// clearmoe_route_noalloc: the routing step for callers that cannot allocate device memory.
//
// Some callers of this library cannot call cudaMalloc: code that runs inside another engine's
// enqueue path (inference-server or plugin hosts that own every device byte and forbid
// allocation there), processes held to a fixed device-memory budget, and latency-critical loops
// where cudaMalloc's implicit device-wide synchronisation is not acceptable. The handle-based
// calls allocate their workspace in clearmoe_layer_create, so this entry point offers the routing
// kernels without a handle: their scratch (the per-range expert histograms and a status word) is a
// file-scope device array that every GPU loading the library holds until the process exits; the
// per-token words of the routing (expert | rank in range) travel through the caller's idx, which
// the finalize kernel then rewrites with the experts alone.
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace {

// Scratch layout (int32 words): [2] status word used when the caller passes no status pointer,
// [16, 16 + MAX_CTAS * CM_MAX_E) the per-range histograms.
constexpr int kNoallocMaxCtas = 1024;
constexpr int kHistOffset = 16;
constexpr int kScratchWords = kHistOffset + kNoallocMaxCtas * CM_MAX_E;  // 65,600 bytes

static __device__ __align__(256) int32_t g_route_scratch[kScratchWords];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int32_t* g_scratch_addr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};

// Once per device, with that device current: the device address of the scratch array. In host
// code the symbol g_route_scratch is only a host-side stand-in, never a device address.
int scratch_for_current_device(int32_t** addr, int* num_sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return CLEARMOE_ECUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return CLEARMOE_EUNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_route_scratch) != cudaSuccess || !p) {
            (void)cudaGetLastError();
            return CLEARMOE_ECUDA;
        }
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
            (void)cudaGetLastError();
            return CLEARMOE_ECUDA;
        }
        g_num_sms[dev] = sms;
        g_scratch_addr[dev] = static_cast<int32_t*>(p);
    }
    *addr = g_scratch_addr[dev];
    *num_sms = g_num_sms[dev];
    return CLEARMOE_OK;
}

inline bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

}  // namespace

extern "C" int clearmoe_route_noalloc(const void* x, int64_t T, int32_t d, int32_t dtype,
                                      const clearmoe_router* router, int32_t E, int32_t* idx,
                                      int32_t* counts, int32_t* offsets, int32_t* perm,
                                      int32_t* status, void* stream) {
    if (!x || !router || !router->W || !router->b || !idx || !counts || !offsets || !perm)
        return CLEARMOE_EINVAL;
    if (T < 1 || T > ((int64_t)1 << 30) || E < 1 || E > CM_MAX_E) return CLEARMOE_EINVAL;
    if (dtype != CLEARMOE_BF16 && dtype != CLEARMOE_F32) return CLEARMOE_EINVAL;
    if (dtype == CLEARMOE_BF16 ? (d < 64 || d % 64 || d > 1024) : (d < 4 || d % 4 || d > 512))
        return CLEARMOE_EUNSUPPORTED;
    if (misaligned(x, 16) || misaligned(router->W, 16) || misaligned(idx, 4) || misaligned(counts, 4) ||
        misaligned(offsets, 4) || misaligned(perm, 4) || (status && misaligned(status, 4)))
        return CLEARMOE_EINVAL;

    int32_t* scratch = nullptr;
    int num_sms = 0;
    int rc = scratch_for_current_device(&scratch, &num_sms);
    if (rc) return rc;
    int grid = 0, chunk = 0;
    const int g = cm::route_grid(T, d, E, dtype, num_sms, &grid, &chunk);
    if (g) return g == -2 ? CLEARMOE_EUNSUPPORTED : CLEARMOE_ECUDA;
    if (grid > kNoallocMaxCtas) return CLEARMOE_EUNSUPPORTED;  // beyond the scratch's capacity

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // Only the spare status word and the caller's status start at zero; the histograms are
    // fully rewritten by every launch before they are read.
    if (cudaMemsetAsync(scratch + 2, 0, sizeof(int32_t), s) != cudaSuccess ||
        (status && cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess)) {
        (void)cudaGetLastError();
        return CLEARMOE_ECUDA;
    }
    cm::RouteArgs a;
    std::memset(&a, 0, sizeof(a));
    a.x = x;
    a.T = T;
    a.d = d;
    a.E = E;
    a.dtype = dtype;
    a.Wg = router->W;
    a.bg = router->b;
    a.idx = idx;
    a.perm = perm;
    a.inv = nullptr;
    a.counts = counts;
    a.offsets = offsets;
    a.cta_counts = scratch + kHistOffset;
    a.tinfo = idx;  // packed words in idx; route_finalize_kernel unpacks them
    a.debug_skip = -1;
    a.wait_limit_ns = 1000000000LL;
    a.status = status ? status : scratch + 2;
    cudaError_t e = cm::launch_route(a, grid, chunk, s);
    if (e == cudaSuccess) e = cm::launch_route_finalize(a, grid, chunk, s);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return CLEARMOE_ECUDA;
    }
    return CLEARMOE_OK;
}
