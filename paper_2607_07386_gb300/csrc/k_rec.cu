// K-REC: fused sparse gated delta recurrence (Eqs. sdm-decay, sdm-write, sdm-read).
//
// For one (b, h) chain, tokens in order t = 0 .. T-1:
//   r_n  = alpha_t * M[I^w_t[n]]                 (decay of the written slots only)
//   v~   = sum_n w_n r_n                         (prediction)
//   M[I^w_t[n]] = R(r_n + beta_t w_n (v_t - v~)) (delta write, storage rounding R)
//   y_t  = R(sum_n rho_n M[I^r_t[n]])            (read of the post-write memory)
// Every step is elementwise along d_v once (idx, w) are fixed, so a chain is split into
// independent d-ranges.  One CTA owns one (chain, d-range): thread (g, c) moves 16-byte
// chunk c of the rows of slot group g (slots n = g, g+G, ...), so a row is read and
// written as coalesced 16-byte vectors.  The prediction and the read are reduced over the
// slot groups with warp shuffles plus one shared-memory pass.  Ordering: the scatter of
// token t completes (block barrier) before any thread gathers for token t+1 or reads token t.
#include "sdm_internal.h"

namespace sdm {

constexpr int REC_MAX_SPT = 4;     // slots per thread per token (k <= 64 needs >= 16 slot groups)

template <class D, int DCH>
__global__ void __launch_bounds__(512) k_recur(const RecArgs a, int nsplit) {
    constexpr int E = D::E;
    extern __shared__ __align__(16) float smR[];   // [2][NW][DCH][E]  partial sums
    const int nthreads = blockDim.x;
    const int NW = nthreads >> 5;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c = tid % DCH;               // chunk within the CTA's d-range
    const int g = tid / DCH;               // slot group
    const int G = nthreads / DCH;
    const int64_t chain = blockIdx.x / nsplit;
    const int split = blockIdx.x - static_cast<int>(chain) * nsplit;
    const int64_t rowbytes = static_cast<int64_t>(a.dv) * D::BYTES;
    const int64_t coff = static_cast<int64_t>(split * DCH + c) * 16;       // byte offset of my chunk in a row
    char* Mb = static_cast<char*>(a.mem) + chain * a.N * rowbytes + coff;
    const char* vb = static_cast<const char*>(a.v) + chain * a.T * rowbytes + coff;
    char* yb = static_cast<char*>(a.y) + chain * a.T * rowbytes + coff;
    float* red = smR;

    for (int t = 0; t < a.T; ++t) {
        const int64_t tok = chain * a.T + t;
        const float alpha = load_elem<D>(a.alpha, tok);
        const float beta = load_elem<D>(a.beta, tok);
        // ---- gather + decay + partial prediction
        float r[REC_MAX_SPT][E];
        float wn[REC_MAX_SPT];
        int64_t ioff[REC_MAX_SPT];
        float part[E];
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < REC_MAX_SPT; ++j) {
            const int n = g + j * G;
            ioff[j] = -1;
            wn[j] = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) r[j][e] = 0.f;
            if (n < a.kw) {
                const int slot = __ldg(a.idx_w + tok * a.kw + n);
                wn[j] = __ldg(a.w_w + tok * a.kw + n);
                if (slot >= 0 && slot < a.N) {
                    ioff[j] = static_cast<int64_t>(slot) * rowbytes;
                    const uint4 m = *reinterpret_cast<const uint4*>(Mb + ioff[j]);
                    float f[E];
                    unpack16<D>(m, f);
#pragma unroll
                    for (int e = 0; e < E; ++e) {
                        r[j][e] = alpha * f[e];
                        part[e] = fmaf(wn[j], r[j][e], part[e]);
                    }
                } else {
                    flag_error(a.err, ERR_BAD_INDEX);
                }
            }
        }
        // ---- reduce the prediction over slot groups: lanes with the same chunk, then warps
#pragma unroll
        for (int e = 0; e < E; ++e)
            for (int off = DCH; off < 32; off <<= 1) part[e] += __shfl_xor_sync(0xffffffffu, part[e], off);
        float* red0 = red;   // buffer 0: prediction
        if (lane < DCH) {
#pragma unroll
            for (int e = 0; e < E; ++e) red0[(warp * DCH + c) * E + e] = part[e];
        }
        __syncthreads();
        float pred[E];
#pragma unroll
        for (int e = 0; e < E; ++e) pred[e] = 0.f;
        for (int w = 0; w < NW; ++w) {
#pragma unroll
            for (int e = 0; e < E; ++e) pred[e] += red0[(w * DCH + c) * E + e];
        }
        // ---- delta write
        float vt[E];
        {
            const uint4 vv = *reinterpret_cast<const uint4*>(vb + t * rowbytes);
            unpack16<D>(vv, vt);
        }
#pragma unroll
        for (int e = 0; e < E; ++e) vt[e] -= pred[e];   // delta = v - v~
#pragma unroll
        for (int j = 0; j < REC_MAX_SPT; ++j) {
            if (ioff[j] >= 0) {
                const float bw = beta * wn[j];
                float o[E];
#pragma unroll
                for (int e = 0; e < E; ++e) o[e] = fmaf(bw, vt[e], r[j][e]);
                *reinterpret_cast<uint4*>(Mb + ioff[j]) = pack16<D>(o);
            }
        }
        __syncthreads();   // every write of token t is visible before the read and the next gather
        // ---- read of the post-write memory
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < REC_MAX_SPT; ++j) {
            const int n = g + j * G;
            if (n < a.kr) {
                const int slot = __ldg(a.idx_r + tok * a.kr + n);
                const float rho = __ldg(a.w_r + tok * a.kr + n);
                if (slot >= 0 && slot < a.N) {
                    const uint4 m = *reinterpret_cast<const uint4*>(Mb + static_cast<int64_t>(slot) * rowbytes);
                    float f[E];
                    unpack16<D>(m, f);
#pragma unroll
                    for (int e = 0; e < E; ++e) part[e] = fmaf(rho, f[e], part[e]);
                } else {
                    flag_error(a.err, ERR_BAD_INDEX);
                }
            }
        }
#pragma unroll
        for (int e = 0; e < E; ++e)
            for (int off = DCH; off < 32; off <<= 1) part[e] += __shfl_xor_sync(0xffffffffu, part[e], off);
        float* red1 = red + NW * DCH * E;   // buffer 1: read
        if (lane < DCH) {
#pragma unroll
            for (int e = 0; e < E; ++e) red1[(warp * DCH + c) * E + e] = part[e];
        }
        __syncthreads();
        if (g == 0) {
            float yv[E];
#pragma unroll
            for (int e = 0; e < E; ++e) yv[e] = 0.f;
            for (int w = 0; w < NW; ++w) {
#pragma unroll
                for (int e = 0; e < E; ++e) yv[e] += red1[(w * DCH + c) * E + e];
            }
            *reinterpret_cast<uint4*>(yb + t * rowbytes) = pack16<D>(yv);
        }
    }
}

template <class D, int DCH>
static cudaError_t launch_rec_typed(const RecArgs& a, int nsplit, int threads, cudaStream_t stream) {
    const size_t sm = static_cast<size_t>(2) * (threads / 32) * DCH * D::E * sizeof(float);
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    k_recur<D, DCH><<<static_cast<unsigned>(chains * nsplit), threads, sm, stream>>>(a, nsplit);
    return cudaGetLastError();
}

template <class D>
static cudaError_t launch_rec_dtype(const RecArgs& a, cudaStream_t stream) {
    const int nch = a.dv * D::BYTES / 16;         // 16-byte chunks per row
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    // d-split: smallest per-CTA range (>= 2 chunks = one 32-byte sector) that still gives
    // a few hundred CTAs; long chains with few heads get the finest split.
    int dch = 1;
    while (dch < 32 && nch % (dch * 2) == 0) dch *= 2;      // largest power-of-two divisor <= 32
    while (dch > 2 && chains * (nch / dch) < 512) dch /= 2;
    const int nsplit = nch / dch;
    const int kmax = a.kw > a.kr ? a.kw : a.kr;
    // enough slot groups that each thread handles <= REC_MAX_SPT slots, and about k groups
    int groups = kmax;
    int threads = groups * dch;
    threads = (threads + 31) / 32 * 32;
    if (threads < 32) threads = 32;
    if (threads > 512) threads = 512;
    while ((threads / dch) * REC_MAX_SPT < kmax && threads < 512) threads += 32;
    switch (dch) {
        case 1: return launch_rec_typed<D, 1>(a, nsplit, threads, stream);
        case 2: return launch_rec_typed<D, 2>(a, nsplit, threads, stream);
        case 4: return launch_rec_typed<D, 4>(a, nsplit, threads, stream);
        case 8: return launch_rec_typed<D, 8>(a, nsplit, threads, stream);
        case 16: return launch_rec_typed<D, 16>(a, nsplit, threads, stream);
        case 32: return launch_rec_typed<D, 32>(a, nsplit, threads, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_recur(int dtype, const RecArgs& a, cudaStream_t stream) {
    return dtype == 0 ? launch_rec_dtype<F32>(a, stream) : launch_rec_dtype<BF16>(a, stream);
}

}  // namespace sdm
