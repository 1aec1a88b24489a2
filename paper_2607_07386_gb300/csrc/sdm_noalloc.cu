// sdm_recur_noalloc: the recurrence of sdm_recur with its hazard table in a fixed,
// statically reserved device array instead of a caller-provided workspace.
//
// Some callers cannot hand the library any device memory: a host runtime whose own pool
// owns the device and exposes no scratch buffers, or a per-token serving loop that must
// not call an allocator (cudaMalloc can synchronise the device and stall every other
// stream in the process).  For them this entry point takes only the tensors of the
// method; the scratch is the file-scope array below, reserved when this module loads.
//
// Limits and behaviour:
//   * the hazard table needs B * H * T * max(k_write, k_read) * 4 bytes; calls that need
//     more than SDM_RECUR_NOALLOC_SCRATCH_BYTES are rejected (SDM_ERR_UNSUPPORTED) before
//     anything is launched;
//   * the array's address is looked up once per device (cudaGetSymbolAddress, with that
//     device current) on the first call made with it current, and cached; that first call
//     therefore does host-side set-up work and should come before any stream capture.  A
//     device reset (cudaDeviceReset) after that first call is not supported: the cached
//     address would outlive the context it belongs to;
//   * every entry of the table that the kernels read is written by the hazard kernel first
//     in the same call, so nothing has to start at zero;
//   * there is one array per device: calls that overlap on the GPU (different streams, or
//     host threads issuing to the same device concurrently) race on it.  Serialise them.
#include "sdm_internal.h"
#include "sdm.h"

#include <stdio.h>

#include <atomic>

namespace {

constexpr size_t kScratchBytes = SDM_RECUR_NOALLOC_SCRATCH_BYTES;
static_assert(kScratchBytes % 256 == 0, "scratch size must be a multiple of 256 bytes");

static __device__ __align__(256) int32_t g_rec_scratch[kScratchBytes / sizeof(int32_t)];

constexpr int kMaxDevices = 64;
std::atomic<int32_t*> g_rec_scratch_addr[kMaxDevices];

sdm_status cuda_error(cudaError_t e, const char* where) {
    char buf[256];
    snprintf(buf, sizeof(buf), "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
    return sdm::api_error(SDM_ERR_CUDA, buf);
}

// Address of g_rec_scratch on the current device (looked up once per device).
sdm_status scratch_address(int32_t** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_error(e, "sdm_recur_noalloc: cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return sdm::api_error(SDM_ERR_UNSUPPORTED, "sdm_recur_noalloc: device ordinal >= 64");
    int32_t* p = g_rec_scratch_addr[dev].load(std::memory_order_acquire);
    if (p == nullptr) {
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_rec_scratch);
        if (e != cudaSuccess) return cuda_error(e, "sdm_recur_noalloc: cudaGetSymbolAddress(scratch)");
        if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 255) != 0)
            return sdm::api_error(SDM_ERR_CUDA, "sdm_recur_noalloc: scratch address is not 256-byte aligned");
        g_rec_scratch_addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return SDM_OK;
}

}  // namespace

extern "C" sdm_status sdm_recur_noalloc(const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                                        const int32_t* idx_r, const float* w_r, const void* v, const void* alpha,
                                        const void* beta, void* mem, void* y, sdm_stream_t stream) {
    if (s == nullptr) return sdm::api_error(SDM_ERR_INVALID_ARG, "sdm_recur_noalloc: shape is NULL");
    // size limit first: it needs no device and rejects before any CUDA call.  The entry
    // count B*H*T*kmax is checked factor by factor against the capacity, so it cannot wrap.
    if (s->B < 0 || s->H < 0 || s->T < 0)
        return sdm::api_error(SDM_ERR_INVALID_ARG, "sdm_recur_noalloc: B, H, T must be >= 0");
    if (s->k_write < 1 || s->k_read < 1 || s->k_write > 64 || s->k_read > 64)
        return sdm::api_error(SDM_ERR_UNSUPPORTED, "sdm_recur_noalloc: k_write and k_read must be in [1, 64]");
    {
        const int64_t cap = static_cast<int64_t>(kScratchBytes / sizeof(int32_t));
        const int64_t factors[4] = {s->B, s->H, s->T, s->k_write > s->k_read ? s->k_write : s->k_read};
        int64_t entries = 1;
        bool fits = true;
        for (int64_t f : factors) {
            if (f == 0) { entries = 0; break; }
            if (entries > cap / f) fits = false;     // entries * f > cap
            if (!fits) break;
            entries *= f;
        }
        if (!fits) {
            char buf[256];
            snprintf(buf, sizeof(buf),
                     "sdm_recur_noalloc: the hazard table does not fit the fixed scratch of %zu bytes "
                     "(B*H*T*max(k_write,k_read) must be <= %lld); use sdm_recur with a workspace",
                     kScratchBytes, static_cast<long long>(cap));
            return sdm::api_error(SDM_ERR_UNSUPPORTED, buf);
        }
    }
    sdm::RecArgs r{};
    bool empty = false;
    sdm_status st = sdm::recur_args("sdm_recur_noalloc", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, &r, &empty);
    if (st != SDM_OK) return st;
    if (empty) return sdm::api_ok();
    int32_t* scratch = nullptr;
    st = scratch_address(&scratch);
    if (st != SDM_OK) return st;
    const cudaError_t e = sdm::launch_recur(s->dtype, r, scratch, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_error(e, "sdm_recur_noalloc: recurrence launch");
    return sdm::api_ok();
}
