// K-INIT: broadcast of the learned initial memory (Sec. 3.1, "Learned Initial State M0").
//   mem[b, h, :, :] = M0[h, :, :] for every sequence b.
// Pure bandwidth: M0 is read once (streaming, evict-first) and each 16-byte vector is
// written B times.  Roofline: (1 + B) * H * N * d_v * elem_bytes bytes of HBM traffic.
#include "sdm_internal.h"

namespace sdm {

constexpr int INIT_THREADS = 256;
constexpr int INIT_UNROLL = 8;

__global__ void __launch_bounds__(INIT_THREADS) k_init_memory(const uint4* __restrict__ M0, uint4* __restrict__ mem,
                                                              int64_t nvec, int B) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * INIT_THREADS;
    int64_t i = static_cast<int64_t>(blockIdx.x) * INIT_THREADS + threadIdx.x;
    for (; i + (INIT_UNROLL - 1) * stride < nvec; i += INIT_UNROLL * stride) {
        uint4 x[INIT_UNROLL];
#pragma unroll
        for (int u = 0; u < INIT_UNROLL; ++u) x[u] = __ldcs(M0 + i + u * stride);
        for (int b = 0; b < B; ++b) {
#pragma unroll
            for (int u = 0; u < INIT_UNROLL; ++u) __stcs(mem + b * nvec + i + u * stride, x[u]);
        }
    }
    for (; i < nvec; i += stride) {
        const uint4 x = __ldcs(M0 + i);
        for (int b = 0; b < B; ++b) __stcs(mem + b * nvec + i, x);
    }
}

cudaError_t launch_init_memory(const void* M0, void* mem, int64_t bytes_per_seq, int B, cudaStream_t stream,
                               int ctas_per_sm) {
    const int64_t nvec = bytes_per_seq / 16;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int64_t want = (nvec + INIT_THREADS * INIT_UNROLL - 1) / (INIT_THREADS * INIT_UNROLL);
    const int64_t cap = static_cast<int64_t>(sms) * ctas_per_sm;   // 8 x 256 threads = a full SM
    const int grid = static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
    // The copy needs no shared memory; asking for the shared-memory-heavy carveout anyway
    // lets an SM hold it beside the addressing kernels (an SM changes its carveout only
    // when idle, so kernels with different carveouts cannot share it).
    cudaError_t e = cudaFuncSetAttribute(k_init_memory, cudaFuncAttributePreferredSharedMemoryCarveout,
                                         cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    k_init_memory<<<grid, INIT_THREADS, 0, stream>>>(reinterpret_cast<const uint4*>(M0), reinterpret_cast<uint4*>(mem),
                                                     nvec, B);
    return cudaGetLastError();
}

}  // namespace sdm
