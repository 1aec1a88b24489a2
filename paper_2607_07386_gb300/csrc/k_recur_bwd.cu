// Backward of the sparse gated delta recurrence with in-place undo (App. A.3,
// "Memory-Efficient Backward").
//
// The forward (k_recur with an undo log) updates the memory in place and records, for every
// token t and write slot n, the row M_{t-1}[I^w_t[n]] its write overwrote.  The backward walks
// the tokens in reverse with the memory at M_t and an fp32 adjoint G = dL/dM_t of the rows
// touched so far (dense [N, d_v] per chain, zero elsewhere).  For L = sum_t <dy_t, y_t>:
//
//   read   y_t = sum_n rho_n M_t[r_n]:   d rho_n = <dy_t, M_t[r_n]>,  G[r_n] += rho_n dy_t
//   write  M_t[i] = r_i + beta w_i delta,  r_i = alpha M_{t-1}[i],  delta = v_t - sum_m w_m r_m:
//          d delta = beta sum_i w_i G_i,  d beta = sum_i w_i <G_i, delta>,
//          d w_i = beta <G_i, delta> - <r_i, d delta>,  d v_t = d delta,
//          d r_i = G_i - w_i d delta,  d alpha = sum_i <d r_i, M_{t-1}[i]>,
//          G[i] <- alpha d r_i,  M[i] <- M_{t-1}[i] (the undo)
//
// Storage rounding of the forward is not differentiated (the rows are the stored values).
// One warp per (b, h) chain; lane l holds elements l, l + 32, ... of every row.  Plain loads
// and stores only: no asynchronous copies and no waits.  The forward kernels' prefetch
// machinery is the next step for this one.
#include "sdm_internal.h"

namespace sdm {

constexpr int BW_WARPS = 4;
constexpr int BW_MAXE = 8;          // d_v <= 256

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
    return x;
}

template <class D> __device__ __forceinline__ void copy_elem(void* dst, const void* src, int64_t i);
template <> __device__ __forceinline__ void copy_elem<F32>(void* dst, const void* src, int64_t i) {
    reinterpret_cast<float*>(dst)[i] = reinterpret_cast<const float*>(src)[i];
}
template <> __device__ __forceinline__ void copy_elem<BF16>(void* dst, const void* src, int64_t i) {
    reinterpret_cast<unsigned short*>(dst)[i] = reinterpret_cast<const unsigned short*>(src)[i];
}

template <class D>
__global__ void __launch_bounds__(32 * BW_WARPS) k_recur_bwd(const RecArgs a, const void* __restrict__ undo,
                                                             const void* __restrict__ dy, float* __restrict__ dv_o,
                                                             float* __restrict__ dalpha, float* __restrict__ dbeta,
                                                             float* __restrict__ dw_w, float* __restrict__ dw_r,
                                                             float* __restrict__ dM) {
    const int lane = threadIdx.x & 31;
    const int64_t chain = static_cast<int64_t>(blockIdx.x) * BW_WARPS + (threadIdx.x >> 5);
    if (chain >= static_cast<int64_t>(a.B) * a.H) return;              // whole warps
    const int dv = a.dv, T = a.T, kw = a.kw, kr = a.kr;
    const int epl = dv / 32;                                             // elements per lane
    const uint32_t N = static_cast<uint32_t>(a.N);
    const int64_t mbase = chain * a.N * dv;                              // element offset of the chain's memory
    float* G = dM + mbase;
    bool bad = false, unsorted = false;
    for (int t = T - 1; t >= 0; --t) {
        const int64_t tok = chain * T + t;
        const float alpha = load_elem<D>(a.alpha, tok), beta = load_elem<D>(a.beta, tok);
        float gy[BW_MAXE];
#pragma unroll
        for (int j = 0; j < BW_MAXE; ++j) gy[j] = j < epl ? load_elem<D>(dy, tok * dv + lane + 32 * j) : 0.f;
        // ---- read of the post-write memory M_t
        for (int n = 0; n < kr; ++n) {
            const int32_t s = __ldg(a.idx_r + tok * kr + n);
            unsorted |= n > 0 && __ldg(a.idx_r + tok * kr + n - 1) >= s;
            if (static_cast<uint32_t>(s) >= N) { bad = true; continue; }   // warp-uniform
            const float rho = __ldg(a.w_r + tok * kr + n);
            const int64_t row = mbase + static_cast<int64_t>(s) * dv;
            float p = 0.f;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    const int64_t e = static_cast<int64_t>(s) * dv + lane + 32 * j;
                    p = fmaf(gy[j], load_elem<D>(a.mem, row + lane + 32 * j), p);
                    G[e] = fmaf(rho, gy[j], G[e]);
                }
            }
            p = warp_sum(p);
            if (lane == 0) dw_r[tok * kr + n] = p;
        }
        // ---- the write: prediction and delta from the logged rows, d delta from the adjoint
        float vt[BW_MAXE], pred[BW_MAXE], dd[BW_MAXE];
#pragma unroll
        for (int j = 0; j < BW_MAXE; ++j) {
            vt[j] = j < epl ? load_elem<D>(a.v, tok * dv + lane + 32 * j) : 0.f;
            pred[j] = 0.f;
            dd[j] = 0.f;
        }
        for (int m = 0; m < kw; ++m) {
            const int32_t i = __ldg(a.idx_w + tok * kw + m);
            // the write slots of a token must be distinct: checked as strictly ascending
            unsorted |= m > 0 && __ldg(a.idx_w + tok * kw + m - 1) >= i;
            if (static_cast<uint32_t>(i) >= N) continue;                // no write, no log entry
            const float w = __ldg(a.w_w + tok * kw + m);
            const int64_t urow = (tok * kw + m) * dv;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    pred[j] = fmaf(w, alpha * load_elem<D>(undo, urow + lane + 32 * j), pred[j]);
                    dd[j] = fmaf(w, G[static_cast<int64_t>(i) * dv + lane + 32 * j], dd[j]);
                }
            }
        }
        float delta[BW_MAXE];
#pragma unroll
        for (int j = 0; j < BW_MAXE; ++j) {
            delta[j] = vt[j] - pred[j];
            dd[j] *= beta;
            if (j < epl) dv_o[tok * dv + lane + 32 * j] = dd[j];
        }
        float db = 0.f, da = 0.f;
        for (int m = 0; m < kw; ++m) {
            const int32_t i = __ldg(a.idx_w + tok * kw + m);
            if (static_cast<uint32_t>(i) >= N) { bad = true; if (lane == 0) dw_w[tok * kw + m] = 0.f; continue; }
            const float w = __ldg(a.w_w + tok * kw + m);
            const int64_t urow = (tok * kw + m) * dv;
            float gd = 0.f, rd = 0.f;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    const int64_t e = static_cast<int64_t>(i) * dv + lane + 32 * j;
                    const float prev = load_elem<D>(undo, urow + lane + 32 * j);
                    const float gi = G[e];
                    gd = fmaf(gi, delta[j], gd);
                    rd = fmaf(alpha * prev, dd[j], rd);
                    const float dr = gi - w * dd[j];
                    da = fmaf(dr, prev, da);
                    G[e] = alpha * dr;
                }
            }
            gd = warp_sum(gd);
            rd = warp_sum(rd);
            db = fmaf(w, gd, db);
            if (lane == 0) dw_w[tok * kw + m] = beta * gd - rd;
        }
        da = warp_sum(da);
        if (lane == 0) { dalpha[tok] = da; dbeta[tok] = db; }
        // ---- undo: M_t -> M_{t-1} on the written rows (after every read of M_t above)
        for (int m = 0; m < kw; ++m) {
            const int32_t i = __ldg(a.idx_w + tok * kw + m);
            if (static_cast<uint32_t>(i) >= N) continue;
            const int64_t urow = (tok * kw + m) * dv;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j)
                if (j < epl) copy_elem<D>(static_cast<char*>(a.mem) + (mbase + static_cast<int64_t>(i) * dv) * D::BYTES,
                                          static_cast<const char*>(undo) + urow * D::BYTES, lane + 32 * j);
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, unsorted) && lane == 0) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_recur_backward(int dtype, const RecArgs& a, const void* undo, const void* dy, float* dv,
                                  float* dalpha, float* dbeta, float* dw_w, float* dw_r, float* dM, cudaStream_t stream) {
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    const unsigned grid = static_cast<unsigned>((chains + BW_WARPS - 1) / BW_WARPS);
    if (dtype == 0)
        k_recur_bwd<F32><<<grid, 32 * BW_WARPS, 0, stream>>>(a, undo, dy, dv, dalpha, dbeta, dw_w, dw_r, dM);
    else
        k_recur_bwd<BF16><<<grid, 32 * BW_WARPS, 0, stream>>>(a, undo, dy, dv, dalpha, dbeta, dw_w, dw_r, dM);
    return cudaGetLastError();
}

}  // namespace sdm
