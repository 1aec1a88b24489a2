// K-LAZY: copy-on-write seeding of the learned initial memory (Sec. 3.1, "Learned Initial
// State M0"), in place of the B-fold broadcast of K-INIT.
//
// The memory of chain c = (b, h) is an overlay: slot s holds a row in mem[c] only once some
// token has written it (bit s of the chain's touched bitmap); until then its value is
// M0[h, s], and mem[c, s] is never read.  Per call (T tokens):
//   k_fw_init    firstw[c][s] = touched(c, s) ? -1 : INT_MAX
//   k_fw_write   firstw[c][s] = min(firstw[c][s], t) for every write entry (t, n) with
//                idx_w[c, t, n] = s
//   k_fw_bitmap  touched(c, s) = (firstw[c][s] != INT_MAX)
// and the hazard pass marks a gather of slot s by token t "fresh" when firstw[c][s] >= t:
// nothing wrote s before token t, in this call or an earlier one, so the row is M0's.  The
// recurrence then gathers that row from M0 instead of mem (a write-gather of a fresh slot
// decays M0's row, Eq. sdm-decay; a read-gather of one reads it, Eq. sdm-read).
// k_materialize turns the overlay into the dense memory of K-INIT + forward by writing
// M0's row into every untouched slot.
//
// Traffic per call: firstw is chains * N * 4 bytes written twice and read once (L2-sized
// at the layer workload: 134 MB), the bitmap chains * N / 8 bytes each way; the write
// entries are read once.  None of it grows with d_v, while the broadcast it replaces moves
// (1 + B) * H * N * d_v * elem_bytes.
#include "sdm_internal.h"

namespace sdm {

constexpr int LZ_THREADS = 256;

// One thread per slot; slots of a chain run over [0, words * 32) so that a warp covers one
// bitmap word.
__global__ void __launch_bounds__(LZ_THREADS) k_fw_init(const uint32_t* __restrict__ touched, int32_t* __restrict__ firstw,
                                                        int64_t chains, uint32_t N, uint32_t words) {
    const int64_t per_chain = static_cast<int64_t>(words) * 32;
    const int64_t total = chains * per_chain;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * LZ_THREADS;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * LZ_THREADS + threadIdx.x; i < total; i += stride) {
        const int64_t c = i / per_chain;
        const uint32_t s = static_cast<uint32_t>(i - c * per_chain);
        if (s >= N) continue;
        const uint32_t w = __ldg(touched + c * words + (s >> 5));
        firstw[c * N + s] = ((w >> (s & 31)) & 1u) ? -1 : INT_MAX;
    }
}

// One thread per write entry of the call's [chains, T, kw] list.
__global__ void __launch_bounds__(LZ_THREADS) k_fw_write(const int32_t* __restrict__ idx_w, int32_t* __restrict__ firstw,
                                                         int64_t entries, int T, int kw, uint32_t N) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * LZ_THREADS;
    const int64_t per_chain = static_cast<int64_t>(T) * kw;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * LZ_THREADS + threadIdx.x; e < entries; e += stride) {
        const int32_t s = __ldg(idx_w + e);
        if (static_cast<uint32_t>(s) >= N) continue;    // invalid slots are reported by the recurrence
        const int64_t c = e / per_chain;
        const int t = static_cast<int>((e - c * per_chain) / kw);
        atomicMin(firstw + c * N + s, t);
    }
}

// One warp per bitmap word: lane l tests slot 32 * word + l.
__global__ void __launch_bounds__(LZ_THREADS) k_fw_bitmap(const int32_t* __restrict__ firstw, uint32_t* __restrict__ touched,
                                                          int64_t chains, uint32_t N, uint32_t words) {
    const int lane = threadIdx.x & 31;
    const int64_t total = chains * words;
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (LZ_THREADS / 32);
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * (LZ_THREADS / 32) + (threadIdx.x >> 5); q < total; q += wstride) {
        const int64_t c = q / words;
        const uint32_t s = static_cast<uint32_t>(q - c * words) * 32 + lane;
        const bool hit = s < N && __ldg(firstw + c * N + s) != INT_MAX;
        const uint32_t word = __ballot_sync(0xffffffffu, hit);
        if (lane == 0) touched[q] = word;
    }
}

// One thread per 16-byte vector of mem; untouched slots receive M0's row.
__global__ void __launch_bounds__(LZ_THREADS) k_materialize(const uint4* __restrict__ M0, const uint32_t* __restrict__ touched,
                                                            uint4* __restrict__ mem, int64_t chains, int H, uint32_t N,
                                                            uint32_t words, uint32_t vpr) {
    const int64_t per_chain = static_cast<int64_t>(N) * vpr;
    const int64_t total = chains * per_chain;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * LZ_THREADS;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * LZ_THREADS + threadIdx.x; i < total; i += stride) {
        const int64_t c = i / per_chain;
        const int64_t r = i - c * per_chain;
        const uint32_t s = static_cast<uint32_t>(r / vpr);
        const uint32_t w = __ldg(touched + c * words + (s >> 5));
        if ((w >> (s & 31)) & 1u) continue;
        mem[i] = __ldg(M0 + static_cast<int64_t>(c % H) * per_chain + r);
    }
}

namespace {
unsigned grid_for(int64_t work, int per_block) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (work + per_block - 1) / per_block;
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * 8;   // 8 x 256 threads fill an SM
    return static_cast<unsigned>(want < 1 ? 1 : (want < cap ? want : cap));
}
}  // namespace

cudaError_t launch_lazy_prepare(const uint32_t* touched, int32_t* firstw, const int32_t* idx_w, int64_t chains, int T,
                                int kw, int64_t N, cudaStream_t stream) {
    const uint32_t n32 = static_cast<uint32_t>(N);
    const uint32_t words = static_cast<uint32_t>((N + 31) / 32);
    k_fw_init<<<grid_for(chains * words * 32, LZ_THREADS), LZ_THREADS, 0, stream>>>(touched, firstw, chains, n32, words);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t entries = chains * T * static_cast<int64_t>(kw);
    k_fw_write<<<grid_for(entries, LZ_THREADS), LZ_THREADS, 0, stream>>>(idx_w, firstw, entries, T, kw, n32);
    return cudaGetLastError();
}

cudaError_t launch_lazy_bitmap(const int32_t* firstw, uint32_t* touched, int64_t chains, int64_t N, cudaStream_t stream) {
    const uint32_t words = static_cast<uint32_t>((N + 31) / 32);
    k_fw_bitmap<<<grid_for(chains * words, LZ_THREADS / 32), LZ_THREADS, 0, stream>>>(firstw, touched, chains,
                                                                                       static_cast<uint32_t>(N), words);
    return cudaGetLastError();
}

cudaError_t launch_materialize(const void* M0, const uint32_t* touched, void* mem, int64_t chains, int H, int64_t N,
                               int64_t rowbytes, cudaStream_t stream) {
    const uint32_t words = static_cast<uint32_t>((N + 31) / 32);
    const uint32_t vpr = static_cast<uint32_t>(rowbytes / 16);
    k_materialize<<<grid_for(chains * N * vpr, LZ_THREADS), LZ_THREADS, 0, stream>>>(
        static_cast<const uint4*>(M0), touched, static_cast<uint4*>(mem), chains, H, static_cast<uint32_t>(N), words, vpr);
    return cudaGetLastError();
}

}  // namespace sdm
