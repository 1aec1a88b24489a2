// K-INIT: broadcast of the learned initial memory (Sec. 3.1, "Learned Initial State M0").
//   mem[b, h, :, :] = M0[h, :, :] for every sequence b.
// Pure bandwidth: M0 is read once and each byte is written B times.  Roofline:
// (1 + B) * H * N * d_v * elem_bytes bytes of HBM traffic.  Two forms: k_init_memory, a
// grid-stride copy by SM threads (sdm_init_memory, the copy alone), and k_init_bulk, a copy
// driven through the bulk-copy engine by one thread per SM (sdm_forward_m0, the copy beside
// the addressing).
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

// The same broadcast through the bulk-copy (TMA) engine, for the copy that runs beside the
// addressing: one thread per CTA, one CTA per SM.  The thread loads 16 KB of M0 into shared
// memory (cp.async.bulk, completion on an mbarrier) and stores that buffer to all B sequences
// (B cp.async.bulk stores, one bulk group), double-buffered: the load of the next chunk goes
// out once the stores of the chunk before have read their buffer.  The copy engine keeps the
// bytes in flight, so the CTA holds one warp, 32 KB of shared memory and few registers, and the
// addressing kernels keep the rest of the SM.
constexpr int IB_CHUNK = 16384;

__device__ __forceinline__ bool ib_wait(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    for (;;) {
        uint32_t done;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(done) : "r"(bar), "r"(parity) : "memory");
        if (done) return true;
        if (clock64() - t0 > 4000000000LL) return false;
    }
}

__global__ void __launch_bounds__(32, 1) k_init_bulk(const char* __restrict__ M0, char* __restrict__ mem,
                                                     int64_t bytes_per_seq, int B, int* err) {
    __shared__ __align__(128) unsigned char buf[2][IB_CHUNK];
    __shared__ __align__(8) unsigned long long bar[2];
    if (threadIdx.x != 0) return;
    const uint32_t sb0 = static_cast<uint32_t>(__cvta_generic_to_shared(buf[0]));    // buffer s at sb0 + s * IB_CHUNK
    const uint32_t mb0 = static_cast<uint32_t>(__cvta_generic_to_shared(&bar[0]));    // barrier s at mb0 + 8 * s
    for (int i = 0; i < 2; ++i) asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(mb0 + 8 * i) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    const int64_t nchunks = (bytes_per_seq + IB_CHUNK - 1) / IB_CHUNK;
    auto load = [&](int64_t c, int s) {
        const int64_t left = bytes_per_seq - c * IB_CHUNK;
        const uint32_t n = static_cast<uint32_t>(left < IB_CHUNK ? left : IB_CHUNK);
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(mb0 + 8 * s), "r"(n) : "memory");
        asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n"
                     ::"r"(sb0 + s * IB_CHUNK), "l"(M0 + c * IB_CHUNK), "r"(n), "r"(mb0 + 8 * s) : "memory");
    };
    bool ok = true;
    int64_t c = blockIdx.x;
    if (c < nchunks) load(c, 0);
    for (int i = 0; c < nchunks; ++i, c += gridDim.x) {
        const int s = i & 1;
        if (!ib_wait(mb0 + 8 * s, static_cast<uint32_t>(i >> 1) & 1u)) { ok = false; break; }
        const int64_t left = bytes_per_seq - c * IB_CHUNK;
        const uint32_t n = static_cast<uint32_t>(left < IB_CHUNK ? left : IB_CHUNK);
        for (int b = 0; b < B; ++b)
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n"
                         ::"l"(mem + b * bytes_per_seq + c * IB_CHUNK), "r"(sb0 + s * IB_CHUNK), "r"(n) : "memory");
        asm volatile("cp.async.bulk.commit_group;\n" ::: "memory");
        if (c + gridDim.x < nchunks) {
            // the other buffer was read by the stores of the chunk before this one
            asm volatile("cp.async.bulk.wait_group.read 1;\n" ::: "memory");
            load(c + gridDim.x, s ^ 1);
        }
    }
    asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory");
    if (!ok) flag_error(err, ERR_TIMEOUT);
}

cudaError_t launch_init_bulk(const void* M0, void* mem, int64_t bytes_per_seq, int B, int* err, cudaStream_t stream) {
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int64_t nchunks = (bytes_per_seq + IB_CHUNK - 1) / IB_CHUNK;
    const unsigned grid = static_cast<unsigned>(nchunks < sms ? (nchunks > 0 ? nchunks : 1) : sms);
    k_init_bulk<<<grid, 32, 0, stream>>>(static_cast<const char*>(M0), static_cast<char*>(mem), bytes_per_seq, B, err);
    return cudaGetLastError();
}

}  // namespace sdm
