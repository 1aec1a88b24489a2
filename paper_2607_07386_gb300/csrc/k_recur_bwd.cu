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
//
// The log can also come back from a quantised snapshot (App. A.3: fp8 or int4 snapshots of
// the log for long sequences): k_undo_quantize codes every logged row with one float32 scale
// s = max|row| / top (448 for e4m3, 7 for int4) and codes round(row / s), all in float32 with
// correctly rounded operations; the backward then takes the logged row as the stored value of
// q * s (rounded to the storage type), for the chain rule and for the undo alike.
// One warp per (b, h) chain; lane l holds elements l, l + 32, ... of every row.  Plain loads
// and stores only: no asynchronous copies and no waits.  The forward kernels' prefetch
// machinery is the next step for this one.
#include "sdm_internal.h"

#include <cuda_fp8.h>

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

// The undo log as the backward reads it: Q = 0 the stored rows themselves; Q = 1 fp8 (e4m3)
// codes, one byte per element; Q = 2 int4 codes, two per byte (element 2i in the low nibble),
// two's complement; one float32 scale per row for Q > 0.
struct UndoLog {
    const void* rows;          // Q = 0: [rows][d_v] storage elements
    const uint8_t* codes;      // Q > 0: [rows][d_v] (fp8) or [rows][d_v / 2] (int4) bytes
    const float* scales;       // Q > 0: [rows]
};

template <class D> __device__ __forceinline__ float to_storage(float x);
template <> __device__ __forceinline__ float to_storage<F32>(float x) { return x; }
template <> __device__ __forceinline__ float to_storage<BF16>(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// Element e of logged row r (a stored value of the storage type D).
template <class D, int Q>
__device__ __forceinline__ float undo_elem(const UndoLog& u, int64_t r, int dv, int e) {
    if constexpr (Q == 0) {
        return load_elem<D>(u.rows, r * dv + e);
    } else if constexpr (Q == 1) {
        const __half_raw hr = __nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(__ldg(u.codes + r * dv + e)), __NV_E4M3);
        return to_storage<D>(__half2float(__half(hr)) * __ldg(u.scales + r));
    } else {
        const int b = __ldg(u.codes + r * (dv / 2) + (e >> 1));
        const int q = (e & 1) ? (static_cast<int>(static_cast<uint32_t>(b) << 24) >> 28)
                              : (static_cast<int>(static_cast<uint32_t>(b) << 28) >> 28);
        return to_storage<D>(static_cast<float>(q) * __ldg(u.scales + r));
    }
}

// Quantised snapshot of the log: one warp per logged row, lane l holding elements l, l + 32, ...
template <class D, int Q>
__global__ void __launch_bounds__(256) k_undo_quantize(const void* __restrict__ undo, int64_t rows, int dv,
                                                       uint8_t* __restrict__ codes, float* __restrict__ scales) {
    const int lane = threadIdx.x & 31;
    const int epl = dv / 32;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; r < rows; r += nwarps) {
        float x[BW_MAXE];
        float am = 0.f;
#pragma unroll
        for (int j = 0; j < BW_MAXE; ++j) {
            x[j] = j < epl ? load_elem<D>(undo, r * dv + lane + 32 * j) : 0.f;
            am = fmaxf(am, fabsf(x[j]));
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, off));
        const float s = am > 0.f ? __fdiv_rn(am, Q == 1 ? 448.f : 7.f) : 1.f;
        if (lane == 0) scales[r] = s;
#pragma unroll
        for (int j = 0; j < BW_MAXE; ++j) {
            if (j < epl) {
                const float y = __fdiv_rn(x[j], s);
                if constexpr (Q == 1) {
                    codes[r * dv + lane + 32 * j] = __nv_cvt_float_to_fp8(y, __NV_SATFINITE, __NV_E4M3);
                } else {
                    const int q = min(max(__float2int_rn(y), -7), 7) & 15;
                    const int hi = __shfl_down_sync(0xffffffffu, q, 1);
                    if ((lane & 1) == 0) codes[r * (dv / 2) + ((lane + 32 * j) >> 1)] = static_cast<uint8_t>(q | (hi << 4));
                }
            }
        }
    }
}

cudaError_t launch_undo_quantize(int dtype, int kind, const void* undo, int64_t rows, int dv, void* codes,
                                 float* scales, cudaStream_t stream) {
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int64_t want = (rows + 7) / 8;                       // 8 warps (rows) per CTA
    const int64_t cap = static_cast<int64_t>(sms) * 8;
    const unsigned grid = static_cast<unsigned>(want < cap ? (want > 0 ? want : 1) : cap);
    uint8_t* c = static_cast<uint8_t*>(codes);
    if (dtype == 0)
        kind == 1 ? k_undo_quantize<F32, 1><<<grid, 256, 0, stream>>>(undo, rows, dv, c, scales)
                  : k_undo_quantize<F32, 2><<<grid, 256, 0, stream>>>(undo, rows, dv, c, scales);
    else
        kind == 1 ? k_undo_quantize<BF16, 1><<<grid, 256, 0, stream>>>(undo, rows, dv, c, scales)
                  : k_undo_quantize<BF16, 2><<<grid, 256, 0, stream>>>(undo, rows, dv, c, scales);
    return cudaGetLastError();
}

template <class D> __device__ __forceinline__ void store_elem(void* dst, int64_t i, float x);
template <> __device__ __forceinline__ void store_elem<F32>(void* dst, int64_t i, float x) { reinterpret_cast<float*>(dst)[i] = x; }
template <> __device__ __forceinline__ void store_elem<BF16>(void* dst, int64_t i, float x) {
    reinterpret_cast<__nv_bfloat16*>(dst)[i] = __float2bfloat16_rn(x);
}

template <class D, int Q>
__global__ void __launch_bounds__(32 * BW_WARPS) k_recur_bwd(const RecArgs a, const UndoLog undo,
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
            const int64_t urow = tok * kw + m;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    pred[j] = fmaf(w, alpha * undo_elem<D, Q>(undo, urow, dv, lane + 32 * j), pred[j]);
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
            const int64_t urow = tok * kw + m;
            float gd = 0.f, rd = 0.f;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    const int64_t e = static_cast<int64_t>(i) * dv + lane + 32 * j;
                    const float prev = undo_elem<D, Q>(undo, urow, dv, lane + 32 * j);
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
            const int64_t urow = tok * kw + m;
            char* mrow = static_cast<char*>(a.mem) + (mbase + static_cast<int64_t>(i) * dv) * D::BYTES;
#pragma unroll
            for (int j = 0; j < BW_MAXE; ++j) {
                if (j < epl) {
                    if constexpr (Q == 0)
                        copy_elem<D>(mrow, static_cast<const char*>(undo.rows) + urow * dv * D::BYTES, lane + 32 * j);
                    else
                        store_elem<D>(mrow, lane + 32 * j, undo_elem<D, Q>(undo, urow, dv, lane + 32 * j));
                }
            }
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, unsorted) && lane == 0) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_recur_backward(int dtype, const RecArgs& a, int kind, const void* undo, const void* codes,
                                  const float* scales, const void* dy, float* dv, float* dalpha, float* dbeta,
                                  float* dw_w, float* dw_r, float* dM, cudaStream_t stream) {
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    const unsigned grid = static_cast<unsigned>((chains + BW_WARPS - 1) / BW_WARPS);
    const UndoLog u{undo, static_cast<const uint8_t*>(codes), scales};
#define SDM_BWD(DT, Q) k_recur_bwd<DT, Q><<<grid, 32 * BW_WARPS, 0, stream>>>(a, u, dy, dv, dalpha, dbeta, dw_w, dw_r, dM)
    if (dtype == 0) {
        if (kind == 0) SDM_BWD(F32, 0); else if (kind == 1) SDM_BWD(F32, 1); else SDM_BWD(F32, 2);
    } else {
        if (kind == 0) SDM_BWD(BF16, 0); else if (kind == 1) SDM_BWD(BF16, 1); else SDM_BWD(BF16, 2);
    }
#undef SDM_BWD
    return cudaGetLastError();
}

}  // namespace sdm
