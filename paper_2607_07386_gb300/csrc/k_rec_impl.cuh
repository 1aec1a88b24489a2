// K-REC: fused sparse gated delta recurrence (Eqs. sdm-decay, sdm-write, sdm-read).
//
// For one (b, h) chain, tokens in order t = 0 .. T-1:
//   r_n  = alpha_t * M[I^w_t[n]]                 (decay of the written slots only)
//   v~   = sum_n w_n r_n                         (prediction)
//   M[I^w_t[n]] = R(r_n + beta_t w_n (v_t - v~)) (delta write, storage rounding R)
//   y_t  = R(sum_n rho_n M[I^r_t[n]])            (read of the post-write memory)
//
// Layout of the work.  Every step is elementwise along d_v once (idx, w) are fixed, so a
// chain is split into independent d-ranges and one warp owns one (chain, d-range): lane
// (g, c) moves 16-byte chunk c of the rows of slots n = g*SPT .. g*SPT+SPT-1, so rows are
// read and written as coalesced 16-byte vectors.  The prediction and the read are reduced
// over the G = 32/DCH slot groups in one interleaved shuffle tree; no block barrier.
//
// Latency hiding.  The addressing does not depend on the memory, so the rows token t+LA
// will gather (write-gather and read-gather) are copied into a shared-memory ring with
// cp.async while token t is processed; slot lists, weights, hazard codes and v are copied
// 2*LA tokens ahead.  Stale prefetched rows (slot written in between; see k_hazard.cu) are
// replaced from a shared ring of the rows written by the last LA+1 tokens; a read of a
// slot written by the same token recomputes the writer's value from the same operands
// (bit-identical) in a second, rarely taken reduction.
#pragma once
#include "sdm_internal.h"

namespace sdm {

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

template <int N>
__device__ __forceinline__ void lds_vec(const int* p, int (&o)[N]) {
    if constexpr (N == 1) {
        o[0] = p[0];
    } else if constexpr (N == 2) {
        const int2 v = *reinterpret_cast<const int2*>(p);
        o[0] = v.x; o[1] = v.y;
    } else {
#pragma unroll
        for (int q = 0; q < N / 4; ++q) {
            const int4 v = *reinterpret_cast<const int4*>(p + 4 * q);
            o[4 * q] = v.x; o[4 * q + 1] = v.y; o[4 * q + 2] = v.z; o[4 * q + 3] = v.w;
        }
    }
}

// Token t's lists in shared memory: iw, ww, ir, wr, hz, each KS words (KS = G * SPT, padded to
// 8 words), then the DCH 16-byte chunks of v_t.
__host__ __device__ constexpr int rec_ks_pad(int ks) { return (ks + 7) / 8 * 8; }
__host__ __device__ inline size_t rec_meta_stride(int ks, int dch) { return static_cast<size_t>(5) * rec_ks_pad(ks) * 4 + dch * 16; }
__host__ __device__ inline size_t rec_smem_bytes(int la, int ks, int dch) {
    return static_cast<size_t>(la) * 2 * ks * dch * 16            // prefetched rows
         + static_cast<size_t>(la + 1) * ks * dch * 16              // rows written lately
         + static_cast<size_t>(2 * la + 1) * rec_meta_stride(ks, dch);
}

template <class D, int DCH, int SPT, int LA>
__global__ void __launch_bounds__(32) k_recur(const RecArgs a, int nsplit, const int32_t* __restrict__ hz, int kmax,
                                              int vec_lists) {
    constexpr int E = D::E;
    constexpr int G = 32 / DCH;
    constexpr int KS = G * SPT;
    constexpr int KP = rec_ks_pad(KS);
    constexpr int MR = 2 * LA + 1;
    extern __shared__ __align__(16) unsigned char smR[];
    uint4* rows = reinterpret_cast<uint4*>(smR);                                  // [LA][2][KS][DCH]
    uint4* wring = rows + LA * 2 * KS * DCH;                                        // [LA+1][KS][DCH]
    unsigned char* meta = reinterpret_cast<unsigned char*>(wring + (LA + 1) * KS * DCH);   // [MR][stride]
    const int meta_stride = static_cast<int>(rec_meta_stride(KS, DCH));

    const int lane = threadIdx.x;
    const int c = lane % DCH;
    const int g = lane / DCH;
    const int kw = a.kw, kr = a.kr;
    const int64_t chain = blockIdx.x / nsplit;
    const int split = blockIdx.x - static_cast<int>(chain) * nsplit;
    const int64_t rowbytes = static_cast<int64_t>(a.dv) * D::BYTES;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;
    char* Mb = static_cast<char*>(a.mem) + chain * a.N * rowbytes + dbyte + c * 16;
    const char* vrange = static_cast<const char*>(a.v) + chain * a.T * rowbytes + dbyte;
    char* yb = static_cast<char*>(a.y) + chain * a.T * rowbytes + dbyte + c * 16;
    const int T = a.T;
    const int64_t tok0 = chain * T;
    const int N = static_cast<int>(a.N);

    auto mptr = [&](int slot) { return reinterpret_cast<int*>(meta + slot * meta_stride); };

    // copy token t's lists (and v chunk) into meta slot t % MR
    auto copy_meta = [&](int t) {
        if (t >= T) return;
        int* dst = mptr(t % MR);
        const int64_t tok = tok0 + t;
        if (vec_lists) {   // k multiple of 4 and 16-byte aligned arrays: 16-byte pieces
            const int qw = kw / 4, qr = kr / 4, qm = kmax / 4;
            for (int p = lane; p < 2 * qw + 2 * qr + qm; p += 32) {
                const void* src;
                int* d;
                if (p < qw) { src = a.idx_w + tok * kw + 4 * p; d = dst + 4 * p; }
                else if (p < 2 * qw) { src = a.w_w + tok * kw + 4 * (p - qw); d = dst + KP + 4 * (p - qw); }
                else if (p < 2 * qw + qr) { src = a.idx_r + tok * kr + 4 * (p - 2 * qw); d = dst + 2 * KP + 4 * (p - 2 * qw); }
                else if (p < 2 * qw + 2 * qr) { src = a.w_r + tok * kr + 4 * (p - 2 * qw - qr); d = dst + 3 * KP + 4 * (p - 2 * qw - qr); }
                else { src = hz + tok * kmax + 4 * (p - 2 * qw - 2 * qr); d = dst + 4 * KP + 4 * (p - 2 * qw - 2 * qr); }
                cp_async16(d, src);
            }
        } else {
            for (int p = lane; p < 2 * kw + 2 * kr + kmax; p += 32) {
                const void* src;
                int* d;
                if (p < kw) { src = a.idx_w + tok * kw + p; d = dst + p; }
                else if (p < 2 * kw) { src = a.w_w + tok * kw + (p - kw); d = dst + KP + (p - kw); }
                else if (p < 2 * kw + kr) { src = a.idx_r + tok * kr + (p - 2 * kw); d = dst + 2 * KP + (p - 2 * kw); }
                else if (p < 2 * kw + 2 * kr) { src = a.w_r + tok * kr + (p - 2 * kw - kr); d = dst + 3 * KP + (p - 2 * kw - kr); }
                else { src = hz + tok * kmax + (p - 2 * kw - 2 * kr); d = dst + 4 * KP + (p - 2 * kw - 2 * kr); }
                cp_async4(d, src);
            }
        }
        if (lane < DCH) cp_async16(reinterpret_cast<unsigned char*>(dst) + 5 * KP * 4 + lane * 16, vrange + t * rowbytes + lane * 16);
    };
    // rows that token t gathers (own slots, own chunk) -> rows slot t % LA
    auto copy_rows = [&](int t) {
        if (t >= T) return;
        const int* m = mptr(t % MR);
        const int slot = t % LA;
        int iw[SPT], ir[SPT];
        lds_vec<SPT>(m + g * SPT, iw);
        lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g * SPT + j;
            if (n < kw && iw[j] >= 0 && iw[j] < N) cp_async16(&rows[((slot * 2 + 0) * KS + n) * DCH + c], Mb + iw[j] * rowbytes);
            if (n < kr && ir[j] >= 0 && ir[j] < N) cp_async16(&rows[((slot * 2 + 1) * KS + n) * DCH + c], Mb + ir[j] * rowbytes);
        }
    };

    // gates: lane i holds token 32 * blk + i; broadcast with a shuffle
    float a_cur = 0.f, b_cur = 0.f, a_nxt = 0.f, b_nxt = 0.f;
    if (lane < T) { a_nxt = load_elem<D>(a.alpha, tok0 + lane); b_nxt = load_elem<D>(a.beta, tok0 + lane); }

    // prologue: lists of tokens [0, LA); then rows of [0, LA) with lists of [LA, 2LA)
    for (int u = 0; u < LA; ++u) copy_meta(u);
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    for (int u = 0; u < LA; ++u) {
        copy_rows(u);
        copy_meta(u + LA);
        cp_async_commit();
    }

    for (int t = 0; t < T; ++t) {
        if ((t & 31) == 0) {
            a_cur = a_nxt; b_cur = b_nxt;
            const int tn = t + 32 + lane;
            if (tn < T) { a_nxt = load_elem<D>(a.alpha, tok0 + tn); b_nxt = load_elem<D>(a.beta, tok0 + tn); }
        }
        const float alpha = __shfl_sync(0xffffffffu, a_cur, t & 31);
        const float beta = __shfl_sync(0xffffffffu, b_cur, t & 31);
        cp_async_wait<LA - 1>();        // own rows of token t and lists of token t+LA have landed
        __syncwarp();                   // ... and everyone's; written ring of earlier tokens visible
        const int* m = mptr(t % MR);
        const int rs = t % LA, wsl = t % (LA + 1);
        int iw[SPT], ir[SPT], hzv[SPT];
        float ww[SPT], wr[SPT];
        lds_vec<SPT>(m + g * SPT, iw);
        lds_vec<SPT>(m + KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(ww));
        lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
        lds_vec<SPT>(m + 3 * KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(wr));
        lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);

        // ---- gathers (stale rows from the ring), decay, partial prediction and partial read
        float r[SPT][E];
        float pp[E], yp[E];
#pragma unroll
        for (int e = 0; e < E; ++e) { pp[e] = 0.f; yp[e] = 0.f; }
        bool fix = false;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g * SPT + j;
            const bool okw = n < kw && iw[j] >= 0 && iw[j] < N;
            const bool okr = n < kr && ir[j] >= 0 && ir[j] < N;
            if ((n < kw && !okw) || (n < kr && !okr)) flag_error(a.err, ERR_BAD_INDEX);
            // entries of unused or invalid slots are never filled: they are not read at all
            uint4 mw = make_uint4(0, 0, 0, 0);
            if (okw) {
                mw = rows[((rs * 2 + 0) * KS + n) * DCH + c];
                const int hw = hzv[j] & 0xffff;
                if (hw) {
                    const int d = (hw - 1) >> 6, np = (hw - 1) & 63;
                    mw = wring[(((t - d) % (LA + 1)) * KS + np) * DCH + c];
                }
            }
            float f[E];
            unpack16<D>(mw, f);
            const float wj = okw ? ww[j] : 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) {
                r[j][e] = alpha * f[e];
                pp[e] = fmaf(wj, r[j][e], pp[e]);
            }
            uint4 mr = make_uint4(0, 0, 0, 0);
            float rho = 0.f;
            if (okr) {
                const int hr = (hzv[j] >> 16) & 0xffff;
                rho = wr[j];
                mr = rows[((rs * 2 + 1) * KS + n) * DCH + c];
                if (hr) {
                    const int d = (hr - 1) >> 6, np = (hr - 1) & 63;
                    if (d > 0) {
                        mr = wring[(((t - d) % (LA + 1)) * KS + np) * DCH + c];
                    } else {
                        fix = true;     // value written by this token: added after the write
                        rho = 0.f;
                        mr = make_uint4(0, 0, 0, 0);
                    }
                }
            }
            unpack16<D>(mr, f);
#pragma unroll
            for (int e = 0; e < E; ++e) yp[e] = fmaf(rho, f[e], yp[e]);
        }
#pragma unroll
        for (int off = DCH; off < 32; off <<= 1) {
#pragma unroll
            for (int e = 0; e < E; ++e) {
                pp[e] += __shfl_xor_sync(0xffffffffu, pp[e], off);
                yp[e] += __shfl_xor_sync(0xffffffffu, yp[e], off);
            }
        }
        // ---- delta = v - v~ and the write
        float delta[E];
        unpack16<D>(*reinterpret_cast<const uint4*>(reinterpret_cast<const unsigned char*>(m) + 5 * KP * 4 + c * 16), delta);
#pragma unroll
        for (int e = 0; e < E; ++e) delta[e] -= pp[e];
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g * SPT + j;
            if (n < kw && iw[j] >= 0 && iw[j] < N) {
                const float bw = beta * ww[j];
                float o[E];
#pragma unroll
                for (int e = 0; e < E; ++e) o[e] = fmaf(bw, delta[e], r[j][e]);
                const uint4 packed = pack16<D>(o);
                *reinterpret_cast<uint4*>(Mb + iw[j] * rowbytes) = packed;
                wring[(wsl * KS + n) * DCH + c] = packed;
            }
        }
        // ---- reads of slots this token wrote (rare): recompute the writer's value
        if (__any_sync(0xffffffffu, fix)) {
            float yc[E];
#pragma unroll
            for (int e = 0; e < E; ++e) yc[e] = 0.f;
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                const int n = g * SPT + j;
                const int hr = (hzv[j] >> 16) & 0xffff;
                if (n < kr && ir[j] >= 0 && ir[j] < N && hr && ((hr - 1) >> 6) == 0) {
                    const int np = (hr - 1) & 63;
                    const int hwn = m[4 * KP + np] & 0xffff;        // the writer's own hazard code
                    uint4 base = rows[((rs * 2 + 1) * KS + n) * DCH + c];   // same prefetch as the writer's
                    if (hwn) {
                        const int d2 = (hwn - 1) >> 6, np2 = (hwn - 1) & 63;
                        base = wring[(((t - d2) % (LA + 1)) * KS + np2) * DCH + c];
                    }
                    float f[E], o[E];
                    unpack16<D>(base, f);
                    const float bw = beta * __int_as_float(m[KP + np]);
#pragma unroll
                    for (int e = 0; e < E; ++e) o[e] = fmaf(bw, delta[e], alpha * f[e]);
                    unpack16<D>(pack16<D>(o), f);
                    const float rho = wr[j];
#pragma unroll
                    for (int e = 0; e < E; ++e) yc[e] = fmaf(rho, f[e], yc[e]);
                }
            }
#pragma unroll
            for (int off = DCH; off < 32; off <<= 1) {
#pragma unroll
                for (int e = 0; e < E; ++e) yc[e] += __shfl_xor_sync(0xffffffffu, yc[e], off);
            }
#pragma unroll
            for (int e = 0; e < E; ++e) yp[e] += yc[e];
        }
        if (g == 0) *reinterpret_cast<uint4*>(yb + t * rowbytes) = pack16<D>(yp);
        // ---- prefetch: rows of token t+LA, lists of token t+2LA (the slot of token t-1)
        copy_rows(t + LA);
        copy_meta(t + 2 * LA);
        cp_async_commit();
    }
    cp_async_wait<0>();
}

template <class D, int DCH, int SPT, int LA>
cudaError_t launch_rec_kernel(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    const size_t smem = rec_smem_bytes(LA, (32 / DCH) * SPT, DCH);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur<D, DCH, SPT, LA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    k_recur<D, DCH, SPT, LA><<<static_cast<unsigned>(chains * p.nsplit), 32, smem, s>>>(a, p.nsplit, hz, p.kmax, vec_lists);
    return cudaGetLastError();
}

template <class D, int DCH, int SPT>
cudaError_t launch_rec_la(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vl, cudaStream_t s) {
    return p.la == 1 ? launch_rec_kernel<D, DCH, SPT, 1>(p, a, hz, vl, s) : launch_rec_kernel<D, DCH, SPT, 4>(p, a, hz, vl, s);
}

template <class D, int DCH>
cudaError_t launch_rec_spt(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vl, cudaStream_t s) {
    switch (p.spt) {
        case 1: return launch_rec_la<D, DCH, 1>(p, a, hz, vl, s);
        case 2: return launch_rec_la<D, DCH, 2>(p, a, hz, vl, s);
        case 4: return launch_rec_la<D, DCH, 4>(p, a, hz, vl, s);
        case 8: return launch_rec_la<D, DCH, 8>(p, a, hz, vl, s);
        default: return cudaErrorInvalidValue;
    }
}

template <class D>
cudaError_t launch_rec_dtype(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vl, cudaStream_t s) {
    switch (p.dch) {
        case 1: return launch_rec_spt<D, 1>(p, a, hz, vl, s);
        case 2: return launch_rec_spt<D, 2>(p, a, hz, vl, s);
        case 4: return launch_rec_spt<D, 4>(p, a, hz, vl, s);
        case 8: return launch_rec_spt<D, 8>(p, a, hz, vl, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace sdm
