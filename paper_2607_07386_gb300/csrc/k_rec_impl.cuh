// K-REC: fused sparse gated delta recurrence (Eqs. sdm-decay, sdm-write, sdm-read).
//
// For one (b, h) chain, tokens in order t = 0 .. T-1:
//   r_n  = alpha_t * M[I^w_t[n]]                 (decay of the written slots only)
//   v~   = sum_n w_n r_n                         (prediction)
//   M[I^w_t[n]] = R(r_n + beta_t w_n (v_t - v~)) (delta write, storage rounding R)
//   y_t  = R(sum_n rho_n M[I^r_t[n]])            (read of the post-write memory)
//
// Layout of the work.  Every step is elementwise along d_v once (idx, w) are fixed, so a
// chain is split into independent d-ranges and a warp works on one (chain, d-range): lane
// (g, c) moves 16-byte chunk c of the rows of slots n = g*SPT .. g*SPT+SPT-1, so rows are
// read and written as coalesced 16-byte vectors.  The prediction and the read are reduced
// over the G = 32/DCH slot groups in one interleaved shuffle tree; no block barrier.
//
// Two kernels: k_recur_tw (k_rec_tw.cuh) for T > 1, where several warps interleave the tokens
// of one (chain, d-range) and rows are prefetched ahead through a shared-memory ring; and
// k_recur_one below for one token per chain (a decode step), which needs no hazard pass.
#pragma once
#include "sdm_internal.h"

namespace sdm {

template <class D, int DCH, int SPT, int W, int P>
cudaError_t launch_rec_tw(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s);


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
// Shared-memory address helpers (32-bit shared-window addresses).
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];\n" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}
__device__ __forceinline__ void sts128(uint32_t addr, const uint4& v, bool pred) {
    if (pred) asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}
// 16-byte async copy global -> shared through L2 only; src_bytes = 0 writes zeros.
__device__ __forceinline__ void cp_async16z(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
// The same for a piece of a memory row; when whole256 (rows a multiple of 256 bytes), L2
// fetches the whole aligned 256-byte region around it.
__device__ __forceinline__ void cp_async16z_row(uint32_t dst, const void* src, int src_bytes, bool whole256) {
    if (whole256)
        asm volatile("cp.async.cg.shared.global.L2::256B [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
    else
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}

// ------------------------------------------------------------------------------------------
// One token per chain (a decode step, T == 1): one warp per (chain, d-range), no look-ahead and
// no hazard pass.  The warp loads the token's lists, finds for every read slot whether the
// token also writes it (binary search in the ascending write list) and, on the lazy memory,
// whether the slot is fresh (first-writer table), then gathers all its write and read rows at
// once, and runs the fused body: decay, prediction, delta write, read of the post-write
// memory.  A read of a slot the token writes recomputes the written value from the same
// operands, bit for bit.
// Shared memory of a warp: lists [5][KP] words (idx_w, w_w, idx_r, w_r, codes) + v chunk,
// then rows [2][KS][DCH] x 16 B.
// ------------------------------------------------------------------------------------------
__host__ __device__ inline size_t one_smem_bytes(int ks, int dch) {
    return (rec_meta_stride(ks, dch) + static_cast<size_t>(2) * ks * dch * 16 + 127) / 128 * 128;
}

template <class D, int DCH, int SPT>
__global__ void __launch_bounds__(32) k_recur_one(const RecArgs a, int nsplit, int kmax, int vec_lists) {
    constexpr int E = D::E;
    constexpr int E2 = E / 2;
    constexpr int G = 32 / DCH;
    constexpr int KS = G * SPT;
    constexpr int KP = rec_ks_pad(KS);
    constexpr uint32_t SLOTB = DCH * 16;
    extern __shared__ __align__(128) unsigned char smO[];
    const int lane = threadIdx.x & 31;
    const int64_t gw = blockIdx.x;
    const uint32_t meta0 = static_cast<uint32_t>(__cvta_generic_to_shared(smO));
    int* m = reinterpret_cast<int*>(smO);
    const uint32_t rows0 = meta0 + static_cast<uint32_t>(rec_meta_stride(KS, DCH));
    const int c = lane % DCH;
    const int g = lane / DCH;
    const int kw = a.kw, kr = a.kr;
    const int64_t chain = gw / nsplit;
    const int split = static_cast<int>(gw - chain * nsplit);
    const uint32_t rowbytes = static_cast<uint32_t>(a.dv) * D::BYTES;
    const bool row256 = rowbytes % 256 == 0;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;
    const char* Mc = static_cast<const char*>(a.mem) + chain * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    char* Mw = const_cast<char*>(Mc);
    const char* M0c = a.M0 ? static_cast<const char*>(a.M0) + (chain % a.H) * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16
                           : Mc;
    char* undo_c = a.undo ? static_cast<char*>(a.undo) + dbyte + c * 16 : nullptr;
    const int64_t tok = chain;                           // T == 1
    const uint32_t N = static_cast<uint32_t>(a.N);

    // ---- lists and v
    if (vec_lists) {
        const int qw = kw / 4, qr = kr / 4;
        for (int p = lane; p < 2 * qw + 2 * qr; p += 32) {
            const char* src;
            uint32_t off;
            if (p < qw) { src = reinterpret_cast<const char*>(a.idx_w + tok * kw) + p * 16; off = p * 16; }
            else if (p < 2 * qw) { src = reinterpret_cast<const char*>(a.w_w + tok * kw) + (p - qw) * 16; off = KP * 4 + (p - qw) * 16; }
            else if (p < 2 * qw + qr) { src = reinterpret_cast<const char*>(a.idx_r + tok * kr) + (p - 2 * qw) * 16; off = 2 * KP * 4 + (p - 2 * qw) * 16; }
            else { src = reinterpret_cast<const char*>(a.w_r + tok * kr) + (p - 2 * qw - qr) * 16; off = 3 * KP * 4 + (p - 2 * qw - qr) * 16; }
            cp_async16z(meta0 + off, src, 16);
        }
    } else {
        for (int p = lane; p < kw; p += 32) { m[p] = __ldg(a.idx_w + tok * kw + p); m[KP + p] = __float_as_int(__ldg(a.w_w + tok * kw + p)); }
        for (int p = lane; p < kr; p += 32) { m[2 * KP + p] = __ldg(a.idx_r + tok * kr + p); m[3 * KP + p] = __float_as_int(__ldg(a.w_r + tok * kr + p)); }
    }
    if (lane < DCH)
        cp_async16z(meta0 + 5 * KP * 4 + lane * 16, static_cast<const char*>(a.v) + tok * static_cast<int64_t>(rowbytes) + dbyte + lane * 16, 16);
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    // ---- hazard words (layout of sdm_internal.h): read slot written by this token (code 1 +
    // its write position), fresh flags
    bool unsorted = false;
    for (int p = lane; p < kmax; p += 32) {
        int code = 0;
        if (p < kr) {
            const int s = m[2 * KP + p];
            unsorted |= p > 0 && m[2 * KP + p - 1] >= s;
            int lo = 0, hi = kw;                           // lower bound of s in the write list
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (m[mid] < s) lo = mid + 1; else hi = mid;
            }
            int rc = (lo < kw && m[lo] == s) ? 1 + lo : 0;
            if (a.firstw && static_cast<uint32_t>(s) < N && __ldg(a.firstw + chain * a.N + s) >= 0) rc |= HZ_R_FRESH >> HZ_R_SHIFT;
            code |= rc << HZ_R_SHIFT;
        }
        if (p < kw) {
            const int s = m[p];
            unsorted |= p > 0 && m[p - 1] >= s;
            if (a.firstw && static_cast<uint32_t>(s) < N && __ldg(a.firstw + chain * a.N + s) >= 0) code |= HZ_W_FRESH;
        }
        m[4 * KP + p] = code;
    }
    __syncwarp();
    // ---- gathers of all write and read rows (zero-filled for invalid slots)
    int iw[SPT], ir[SPT], hzv[SPT];
    float ww[SPT], wr[SPT];
    lds_vec<SPT>(m + g * SPT, iw);
    lds_vec<SPT>(m + KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(ww));
    lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
    lds_vec<SPT>(m + 3 * KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(wr));
    lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);
    bool okw[SPT], okr[SPT], bad = false, fix = false;
    const uint32_t my_rows = rows0 + (g * SPT * DCH + c) * 16;
#pragma unroll
    for (int j = 0; j < SPT; ++j) {
        const bool mw = g * SPT + j < kw, mr = g * SPT + j < kr;
        okw[j] = mw && static_cast<uint32_t>(iw[j]) < N;
        okr[j] = mr && static_cast<uint32_t>(ir[j]) < N;
        bad |= (mw && !okw[j]) || (mr && !okr[j]);
        const char* bw = (hzv[j] & HZ_W_FRESH) ? M0c : Mc;
        const char* br = (hzv[j] & HZ_R_FRESH) ? M0c : Mc;
        cp_async16z_row(my_rows + j * SLOTB, bw + static_cast<uint64_t>(okw[j] ? iw[j] : 0) * rowbytes, okw[j] ? 16 : 0, row256);
        cp_async16z_row(my_rows + (KS + j) * SLOTB, br + static_cast<uint64_t>(okr[j] ? ir[j] : 0) * rowbytes, okr[j] ? 16 : 0, row256);
        fix |= okr[j] && hz_rcode(hzv[j]) != 0;
    }
    cp_async_commit();
    const float alpha = load_elem<D>(a.alpha, tok), beta = load_elem<D>(a.beta, tok);
    cp_async_wait<0>();
    __syncwarp();
    // ---- decay, prediction and read partial sums (packed fp32x2 math)
    float2 r[SPT][E2];
    float2 pp[E2], yp[E2];
#pragma unroll
    for (int e = 0; e < E2; ++e) { pp[e] = make_float2(0.f, 0.f); yp[e] = make_float2(0.f, 0.f); }
    const float2 alpha2 = make_float2(alpha, alpha);
#pragma unroll
    for (int j = 0; j < SPT; ++j) {
        const bool rfix = okr[j] && hz_rcode(hzv[j]) != 0;
        const uint4 mwv = lds128(my_rows + j * SLOTB);
        if (undo_c && okw[j]) *reinterpret_cast<uint4*>(undo_c + (tok * kw + g * SPT + j) * static_cast<int64_t>(rowbytes)) = mwv;
        const uint4 mrv = lds128(my_rows + (KS + j) * SLOTB);
        float2 f[E2], h[E2];
        unpack16x2<D>(mwv, f);
        unpack16x2<D>(mrv, h);
        const float wj = okw[j] ? ww[j] : 0.f;
        const float rho = (okr[j] && !rfix) ? wr[j] : 0.f;
        const float2 wj2 = make_float2(wj, wj), rho2 = make_float2(rho, rho);
#pragma unroll
        for (int e = 0; e < E2; ++e) {
            r[j][e] = __fmul2_rn(alpha2, f[e]);
            pp[e] = __ffma2_rn(wj2, r[j][e], pp[e]);
            yp[e] = __ffma2_rn(rho2, h[e], yp[e]);
        }
    }
#pragma unroll
    for (int off = DCH; off < 32; off <<= 1) {
#pragma unroll
        for (int e = 0; e < E2; ++e) {
            const float2 qp = make_float2(__shfl_xor_sync(0xffffffffu, pp[e].x, off), __shfl_xor_sync(0xffffffffu, pp[e].y, off));
            const float2 qy = make_float2(__shfl_xor_sync(0xffffffffu, yp[e].x, off), __shfl_xor_sync(0xffffffffu, yp[e].y, off));
            pp[e] = __fadd2_rn(pp[e], qp);
            yp[e] = __fadd2_rn(yp[e], qy);
        }
    }
    // ---- delta = v - v~ and the write
    float2 d2[E2];
    unpack16x2<D>(lds128(meta0 + 5 * KP * 4 + c * 16), d2);
#pragma unroll
    for (int e = 0; e < E2; ++e) d2[e] = __fadd2_rn(d2[e], make_float2(-pp[e].x, -pp[e].y));
#pragma unroll
    for (int j = 0; j < SPT; ++j) {
        const float bw = beta * ww[j];
        const float2 bw2 = make_float2(bw, bw);
        float2 o[E2];
#pragma unroll
        for (int e = 0; e < E2; ++e) o[e] = __ffma2_rn(bw2, d2[e], r[j][e]);
        if (okw[j]) *reinterpret_cast<uint4*>(Mw + static_cast<uint64_t>(iw[j]) * rowbytes) = pack16x2<D>(o);
    }
    // ---- reads of slots this token wrote: recompute the writer's value from the writer's row
    if (__any_sync(0xffffffffu, fix)) {
        float delta[E];
#pragma unroll
        for (int e = 0; e < E2; ++e) { delta[2 * e] = d2[e].x; delta[2 * e + 1] = d2[e].y; }
        float yc[E];
#pragma unroll
        for (int e = 0; e < E; ++e) yc[e] = 0.f;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int hr = okr[j] ? hz_rcode(hzv[j]) : 0;
            if (hr != 0) {
                const int np = hr - 1;
                float f[E], o[E];
                unpack16<D>(lds128(rows0 + (np * DCH + c) * 16), f);
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
        for (int e = 0; e < E2; ++e) yp[e] = __fadd2_rn(yp[e], make_float2(yc[2 * e], yc[2 * e + 1]));
    }
    if (g == 0)
        *reinterpret_cast<uint4*>(static_cast<char*>(a.y) + tok * static_cast<int64_t>(rowbytes) + dbyte + c * 16) = pack16x2<D>(yp);
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, unsorted) && lane == 0) flag_error(a.err, ERR_UNSORTED);
}

template <class D, int DCH, int SPT>
cudaError_t launch_rec_one(const RecPlan& p, const RecArgs& a, int vec_lists, cudaStream_t s) {
    const size_t smem = one_smem_bytes((32 / DCH) * SPT, DCH);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur_one<D, DCH, SPT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t warps = static_cast<int64_t>(a.B) * a.H * p.nsplit;
    k_recur_one<D, DCH, SPT><<<static_cast<unsigned>(warps), 32, smem, s>>>(a, p.nsplit, p.kmax, vec_lists);
    return cudaGetLastError();
}

template <class D, int DCH, int SPT>
cudaError_t launch_rec_la(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vl, cudaStream_t s) {
    // one token per chain: the single-warp kernel (no look-ahead); otherwise W warps per CTA
    // interleave the tokens of one (chain, d-range)
    if (p.w == 0) return launch_rec_one<D, DCH, SPT>(p, a, vl, s);
    return p.w == 8 ? launch_rec_tw<D, DCH, SPT, 8, 2>(p, a, hz, vl, s) : launch_rec_tw<D, DCH, SPT, 4, 2>(p, a, hz, vl, s);
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

#include "k_rec_tw.cuh"
