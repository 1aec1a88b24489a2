// Access diagnostics of a call's slot selection (App. "Memory Utilization and Access"):
// per token and side, with p the k selected (post-softmax) weights,
//   u(p) = exp(H(p)) / k,  H(p) = -sum_i p_i log p_i     (normalised effective keys)
//   C(m) = p_(1) + ... + p_(m),  p_(1) >= ... >= p_(k)   (cumulative mass of the top m)
// summed over all tokens, plus the number of distinct slots each chain writes and reads.
//
// k_stats_tokens: one warp per (side, token); lane l holds weights l and l + 32 (k <= 64),
// sorts the 64 values descending with a bitonic network across the warp (shuffles), takes
// the inclusive prefix sum, and accumulates u and C(m) in float64 registers over its
// grid-stride items; the selected slots set bits in one bitmap per chain and side.
// k_stats_popc: population count of the bitmaps.
#include "sdm_internal.h"

namespace sdm {

constexpr int ST_THREADS = 256;

__device__ __forceinline__ void cmp_swap_desc(float& a, float& b, bool desc) {
    const float hi = fmaxf(a, b), lo = fminf(a, b);
    a = desc ? hi : lo;
    b = desc ? lo : hi;
}

__global__ void __launch_bounds__(ST_THREADS) k_stats_tokens(const int32_t* __restrict__ idx_w, const float* __restrict__ w_w,
                                                             const int32_t* __restrict__ idx_r, const float* __restrict__ w_r,
                                                             int64_t tokens, int T, int kw, int kr, uint32_t N,
                                                             uint32_t words, uint32_t* __restrict__ bits_w,
                                                             uint32_t* __restrict__ bits_r, double* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int64_t items = 2 * tokens;
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (ST_THREADS / 32);
    double u_w = 0.0, u_r = 0.0;                          // sums of u(p), write and read side
    double cw0 = 0.0, cw1 = 0.0, cr0 = 0.0, cr1 = 0.0;    // sums of C(lane + 1) and C(lane + 33)
    for (int64_t it = static_cast<int64_t>(blockIdx.x) * (ST_THREADS / 32) + (threadIdx.x >> 5); it < items; it += wstride) {
        const int side = static_cast<int>(it & 1);            // 0 = write, 1 = read
        const int64_t tok = it >> 1;
        const int k = side ? kr : kw;
        const int32_t* ix = (side ? idx_r : idx_w) + tok * k;
        const float* wp = (side ? w_r : w_w) + tok * k;
        uint32_t* bits = (side ? bits_r : bits_w) + (tok / T) * words;
        float v0 = -1.f, v1 = -1.f;                          // padding sorts last
        if (lane < k) {
            v0 = __ldg(wp + lane);
            const int32_t s = __ldg(ix + lane);
            if (static_cast<uint32_t>(s) < N) atomicOr(bits + (s >> 5), 1u << (s & 31));
        }
        if (lane + 32 < k) {
            v1 = __ldg(wp + lane + 32);
            const int32_t s = __ldg(ix + lane + 32);
            if (static_cast<uint32_t>(s) < N) atomicOr(bits + (s >> 5), 1u << (s & 31));
        }
        // entropy of the selected weights (0 log 0 = 0)
        float h = (v0 > 0.f ? -v0 * logf(v0) : 0.f) + (v1 > 0.f ? -v1 * logf(v1) : 0.f);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) h += __shfl_xor_sync(0xffffffffu, h, off);
        const double u = static_cast<double>(expf(h)) / k;
        // bitonic sort of the 64 values (element e = lane + 32 r), descending
#pragma unroll
        for (int size = 2; size <= 64; size <<= 1) {
#pragma unroll
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                if (stride == 32) {
                    cmp_swap_desc(v0, v1, true);             // size == 64: elements lane, lane + 32
                } else {
                    const float p0 = __shfl_xor_sync(0xffffffffu, v0, stride);
                    const float p1 = __shfl_xor_sync(0xffffffffu, v1, stride);
                    const bool lower = (lane & stride) == 0;
                    const bool desc0 = (lane & size) == 0;              // element lane
                    const bool desc1 = ((lane + 32) & size) == 0;       // element lane + 32
                    v0 = (lower == desc0) ? fmaxf(v0, p0) : fminf(v0, p0);
                    v1 = (lower == desc1) ? fmaxf(v1, p1) : fminf(v1, p1);
                }
            }
        }
        // inclusive prefix sums: C(lane + 1) over the first 32, C(lane + 33) over the rest
        float c0 = fmaxf(v0, 0.f), c1 = fmaxf(v1, 0.f);
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float q0 = __shfl_up_sync(0xffffffffu, c0, off);
            const float q1 = __shfl_up_sync(0xffffffffu, c1, off);
            if (lane >= off) { c0 += q0; c1 += q1; }
        }
        c1 += __shfl_sync(0xffffffffu, c0, 31);
        const double a0 = lane < k ? static_cast<double>(c0) : 0.0;
        const double a1 = lane + 32 < k ? static_cast<double>(c1) : 0.0;
        if (side) { u_r += u; cr0 += a0; cr1 += a1; }
        else { u_w += u; cw0 += a0; cw1 += a1; }
    }
    // out: [0] u write, [1] u read, [2] unique write, [3] unique read, [4, 4 + kw) C_w, then C_r
    if (lane == 0) {
        atomicAdd(out + 0, u_w);
        atomicAdd(out + 1, u_r);
    }
    if (lane < kw) atomicAdd(out + 4 + lane, cw0);
    if (lane + 32 < kw) atomicAdd(out + 4 + lane + 32, cw1);
    if (lane < kr) atomicAdd(out + 4 + kw + lane, cr0);
    if (lane + 32 < kr) atomicAdd(out + 4 + kw + lane + 32, cr1);
}

__global__ void __launch_bounds__(ST_THREADS) k_stats_popc(const uint32_t* __restrict__ bits_w, const uint32_t* __restrict__ bits_r,
                                                           int64_t nwords, double* __restrict__ out) {
    unsigned long long cw = 0, cr = 0;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * ST_THREADS;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * ST_THREADS + threadIdx.x; i < nwords; i += stride) {
        cw += __popc(__ldg(bits_w + i));
        cr += __popc(__ldg(bits_r + i));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        cw += __shfl_xor_sync(0xffffffffu, cw, off);
        cr += __shfl_xor_sync(0xffffffffu, cr, off);
    }
    if ((threadIdx.x & 31) == 0) {
        atomicAdd(out + 2, static_cast<double>(cw));
        atomicAdd(out + 3, static_cast<double>(cr));
    }
}

cudaError_t launch_access_stats(const int32_t* idx_w, const float* w_w, const int32_t* idx_r, const float* w_r,
                                int64_t chains, int T, int kw, int kr, int64_t N, uint32_t* bits, double* out,
                                cudaStream_t stream) {
    const uint32_t words = static_cast<uint32_t>((N + 31) / 32);
    const int64_t nwords = chains * words;
    cudaError_t e = cudaMemsetAsync(bits, 0, static_cast<size_t>(2 * nwords) * 4, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(out, 0, static_cast<size_t>(4 + kw + kr) * sizeof(double), stream);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t tokens = chains * T;
    const int64_t warps_wanted = 2 * tokens;
    int64_t grid = (warps_wanted + ST_THREADS / 32 - 1) / (ST_THREADS / 32);
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * 8;
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    k_stats_tokens<<<static_cast<unsigned>(grid), ST_THREADS, 0, stream>>>(idx_w, w_w, idx_r, w_r, tokens, T, kw, kr,
                                                                          static_cast<uint32_t>(N), words, bits,
                                                                          bits + nwords, out);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int64_t g2 = (nwords + ST_THREADS - 1) / ST_THREADS;
    if (g2 > cap) g2 = cap;
    if (g2 < 1) g2 = 1;
    k_stats_popc<<<static_cast<unsigned>(g2), ST_THREADS, 0, stream>>>(bits, bits + nwords, nwords, out);
    return cudaGetLastError();
}

}  // namespace sdm
