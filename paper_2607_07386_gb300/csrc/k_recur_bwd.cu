// Backward of the sparse gated delta recurrence with in-place undo (App. A.3,
// "Memory-Efficient Backward").
//
// The forward (the recurrence kernels with an undo log) updates the memory in place and records, for every
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
//
// Layout of the work: one CTA per chain, one warp per 32-element slice of d_v (see k_recur_bwd
// below).  Plain loads and stores, one block barrier per token, no waits on other CTAs.
#include "sdm_internal.h"

#include <cuda_fp8.h>

namespace sdm {

constexpr int BW_MAXE = 8;          // d_v <= 256: elements per lane in the one-warp-per-row passes

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

// One CTA per (b, h) chain, one warp per 32-element slice of d_v (lane l of warp w holds
// element 32 w + l of every row).  Every per-element quantity of the chain rule (the rows of M,
// of G and of the log, pred, delta, d delta, d r) stays in its lane, so the slices walk the
// tokens independently; only the dot products over d_v (d rho, <G_i, delta>, <r_i, d delta>,
// <d r_i, M_{t-1}[i]>) need the slices together.  Each warp reduces its 32 lanes' terms of the
// k_r + 2 k_w products with one butterfly reduce-scatter (lane n ends with the slice's share
// of product n), writes the shares to shared memory, and after one barrier per token warp 0
// adds the slices' shares in slice order and writes dw_r, dw_w, dalpha, dbeta (double-buffered
// by token parity, so one barrier per token suffices).  Row loads of a phase are issued
// together (32 independent loads per lane) before any is used.
constexpr int BW_K = 32;           // slots per list handled by the register batches (k <= 32)

// Butterfly reduce-scatter of 32 per-lane vectors x[0..31] over the warp: afterwards lane n
// holds sum over lanes of x[n] in x[0].
__device__ __forceinline__ void reduce_scatter32(float (&x)[32], int lane) {
#pragma unroll
    for (int lvl = 0; lvl < 5; ++lvl) {
        const int half = 16 >> lvl;              // values kept after this level: half
        const bool upper = (lane >> (4 - lvl)) & 1;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            if (i < half) {
                const float send = upper ? x[i] : x[i + half];
                const float keep = upper ? x[i + half] : x[i];
                x[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16 >> lvl);
            }
        }
    }
}

template <class D, int Q>
__global__ void __launch_bounds__(32 * 8) k_recur_bwd(const RecArgs a, const UndoLog undo,
                                                      const void* __restrict__ dy, float* __restrict__ dv_o,
                                                      float* __restrict__ dalpha, float* __restrict__ dbeta,
                                                      float* __restrict__ dw_w, float* __restrict__ dw_r,
                                                      float* __restrict__ dM) {
    // shares [parity][slice][3 * BW_K + 1]: d rho (k_r), <G, delta> (k_w), <r, dd> (k_w), d alpha
    __shared__ float sh[2][8][3 * BW_K + 1];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nsl = blockDim.x >> 5;
    const int64_t chain = blockIdx.x;
    const int dv = a.dv, T = a.T, kw = a.kw, kr = a.kr;
    const int e = w * 32 + lane;                                         // this lane's element
    const uint32_t N = static_cast<uint32_t>(a.N);
    const int64_t mbase = chain * a.N * dv;
    float* G = dM + mbase;
    char* memc = static_cast<char*>(a.mem) + mbase * D::BYTES;
    bool bad = false, unsorted = false;
    for (int t = T - 1, par = 0; t >= 0; --t, par ^= 1) {
        const int64_t tok = chain * T + t;
        const float alpha = load_elem<D>(a.alpha, tok), beta = load_elem<D>(a.beta, tok);
        const float gy = load_elem<D>(dy, tok * dv + e);
        const float vt = load_elem<D>(a.v, tok * dv + e);
        // lists: lane n holds entry n
        const int32_t ir_l = lane < kr ? __ldg(a.idx_r + tok * kr + lane) : 0;
        const float wr_l = lane < kr ? __ldg(a.w_r + tok * kr + lane) : 0.f;
        const int32_t iw_l = lane < kw ? __ldg(a.idx_w + tok * kw + lane) : 0;
        const float ww_l = lane < kw ? __ldg(a.w_w + tok * kw + lane) : 0.f;
        {
            const int32_t pr = __shfl_up_sync(0xffffffffu, ir_l, 1), pw = __shfl_up_sync(0xffffffffu, iw_l, 1);
            unsorted |= (lane > 0 && lane < kr && pr >= ir_l) || (lane > 0 && lane < kw && pw >= iw_l);
            bad |= (lane < kr && static_cast<uint32_t>(ir_l) >= N) || (lane < kw && static_cast<uint32_t>(iw_l) >= N);
        }
        // ---- read of the post-write memory M_t: d rho_n = <dy, M_t[r_n]>, G[r_n] += rho_n dy
        float x[32];
#pragma unroll
        for (int n = 0; n < BW_K; ++n) {
            const int32_t sn = __shfl_sync(0xffffffffu, ir_l, n);
            const bool ok = n < kr && static_cast<uint32_t>(sn) < N;
            x[n] = ok ? load_elem<D>(memc, static_cast<int64_t>(sn) * dv + e) : 0.f;
        }
        float gr[32];
#pragma unroll
        for (int n = 0; n < BW_K; ++n) {
            const int32_t sn = __shfl_sync(0xffffffffu, ir_l, n);
            gr[n] = (n < kr && static_cast<uint32_t>(sn) < N) ? G[static_cast<int64_t>(sn) * dv + e] : 0.f;
        }
#pragma unroll
        for (int n = 0; n < BW_K; ++n) {
            const int32_t sn = __shfl_sync(0xffffffffu, ir_l, n);
            const float rho = __shfl_sync(0xffffffffu, wr_l, n);
            if (n < kr && static_cast<uint32_t>(sn) < N) G[static_cast<int64_t>(sn) * dv + e] = fmaf(rho, gy, gr[n]);
            x[n] *= gy;
        }
        reduce_scatter32(x, lane);
        sh[par][w][lane] = x[0];                                          // share of d rho_lane
        // ---- the write: prediction and delta from the logged rows, d delta from the adjoint
        float pv[32], gv[32];
#pragma unroll
        for (int m = 0; m < BW_K; ++m) {
            const int32_t im = __shfl_sync(0xffffffffu, iw_l, m);
            const bool ok = m < kw && static_cast<uint32_t>(im) < N;
            pv[m] = ok ? undo_elem<D, Q>(undo, tok * kw + m, dv, e) : 0.f;
            gv[m] = ok ? G[static_cast<int64_t>(im) * dv + e] : 0.f;
        }
        float pred = 0.f, dd = 0.f;
#pragma unroll
        for (int m = 0; m < BW_K; ++m) {
            const float wm = __shfl_sync(0xffffffffu, ww_l, m);
            pred = fmaf(wm, alpha * pv[m], pred);
            dd = fmaf(wm, gv[m], dd);
        }
        const float delta = vt - pred;
        dd *= beta;
        dv_o[tok * dv + e] = dd;
        float gd[32], rd[32], da = 0.f;
#pragma unroll
        for (int m = 0; m < BW_K; ++m) {
            const int32_t im = __shfl_sync(0xffffffffu, iw_l, m);
            const float wm = __shfl_sync(0xffffffffu, ww_l, m);
            const bool ok = m < kw && static_cast<uint32_t>(im) < N;
            gd[m] = gv[m] * delta;
            rd[m] = alpha * pv[m] * dd;
            const float dr = gv[m] - wm * dd;
            da = fmaf(dr, pv[m], da);
            if (ok) {
                G[static_cast<int64_t>(im) * dv + e] = alpha * dr;
                store_elem<D>(memc, static_cast<int64_t>(im) * dv + e, pv[m]);     // the undo
            }
        }
        reduce_scatter32(gd, lane);
        reduce_scatter32(rd, lane);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) da += __shfl_xor_sync(0xffffffffu, da, off);
        sh[par][w][BW_K + lane] = gd[0];
        sh[par][w][2 * BW_K + lane] = rd[0];
        if (lane == 0) sh[par][w][3 * BW_K] = da;
        __syncthreads();
        if (w == 0) {
            float r = 0.f, g = 0.f, q = 0.f, al = 0.f;
            for (int s2 = 0; s2 < nsl; ++s2) {                         // slices in order
                r += sh[par][s2][lane];
                g += sh[par][s2][BW_K + lane];
                q += sh[par][s2][2 * BW_K + lane];
                al += sh[par][s2][3 * BW_K];
            }
            if (lane < kr) dw_r[tok * kr + lane] = r;
            const bool okw = lane < kw && static_cast<uint32_t>(iw_l) < N;
            if (lane < kw) dw_w[tok * kw + lane] = okw ? beta * g - q : 0.f;
            float db = okw ? ww_l * g : 0.f;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) db += __shfl_xor_sync(0xffffffffu, db, off);
            if (lane == 0) { dalpha[tok] = al; dbeta[tok] = db; }
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, unsorted) && lane == 0) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_recur_backward(int dtype, const RecArgs& a, int kind, const void* undo, const void* codes,
                                  const float* scales, const void* dy, float* dv, float* dalpha, float* dbeta,
                                  float* dw_w, float* dw_r, float* dM, cudaStream_t stream) {
    if (a.kw > BW_K || a.kr > BW_K || a.dv % 32 != 0 || a.dv > 256) return cudaErrorInvalidValue;
    const unsigned grid = static_cast<unsigned>(static_cast<int64_t>(a.B) * a.H);
    const int threads = a.dv;                       // one warp per 32-element slice
    const UndoLog u{undo, static_cast<const uint8_t*>(codes), scales};
#define SDM_BWD(DT, Q) k_recur_bwd<DT, Q><<<grid, threads, 0, stream>>>(a, u, dy, dv, dalpha, dbeta, dw_w, dw_r, dM)
    if (dtype == 0) {
        if (kind == 0) SDM_BWD(F32, 0); else if (kind == 1) SDM_BWD(F32, 1); else SDM_BWD(F32, 2);
    } else {
        if (kind == 0) SDM_BWD(BF16, 0); else if (kind == 1) SDM_BWD(BF16, 1); else SDM_BWD(BF16, 2);
    }
#undef SDM_BWD
    return cudaGetLastError();
}

}  // namespace sdm
