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

// Shared memory of one warp of k_recur, rounded so that consecutive warps' regions stay aligned.
__host__ __device__ inline size_t rec_warp_smem_bytes(int la, int ks, int dch) {
    return (rec_smem_bytes(la, ks, dch) + 127) / 128 * 128;
}

// One warp per (chain, d-range); a CTA holds blockDim.x / 32 consecutive warps (the d-ranges
// of one chain when it holds nsplit of them), each with its own shared-memory region.
template <class D, int DCH, int SPT, int LA>
__global__ void __launch_bounds__(256) k_recur(const RecArgs a, int nsplit, const int32_t* __restrict__ hz, int kmax,
                                               int vec_lists) {
    constexpr int E = D::E;
    constexpr int E2 = E / 2;
    constexpr int G = 32 / DCH;
    constexpr int KS = G * SPT;
    constexpr int KP = rec_ks_pad(KS);
    constexpr int MR = 2 * LA + 1;
    constexpr int RING = LA + 1;
    constexpr uint32_t SLOTB = DCH * 16;                 // bytes of one slot's d-range in a ring
    extern __shared__ __align__(128) unsigned char smR[];
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;                                        // warp in the CTA
    const int64_t gw = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + wib;
    if (gw >= static_cast<int64_t>(a.B) * a.H * nsplit) return;              // whole warps
    const uint32_t smbase = static_cast<uint32_t>(__cvta_generic_to_shared(smR));
    const uint32_t sm0 = smbase + wib * static_cast<uint32_t>(rec_warp_smem_bytes(LA, KS, DCH));
    const uint32_t rows0 = sm0;                                              // [LA][2][KS][DCH] x 16 B
    const uint32_t wring0 = rows0 + LA * 2 * KS * SLOTB;                     // [RING][KS][DCH] x 16 B
    const uint32_t meta0 = wring0 + RING * KS * SLOTB;                       // [MR][stride]
    unsigned char* meta_gen = smR + (meta0 - smbase);
    const int meta_stride = static_cast<int>(rec_meta_stride(KS, DCH));

    const int c = lane % DCH;
    const int g = lane / DCH;
    const int kw = a.kw, kr = a.kr;
    const int64_t chain = gw / nsplit;
    const int split = static_cast<int>(gw - chain * nsplit);
    const uint32_t rowbytes = static_cast<uint32_t>(a.dv) * D::BYTES;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;
    const char* Mc = static_cast<const char*>(a.mem) + chain * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    char* Mw = const_cast<char*>(Mc);
    // fresh slots (lazy initial memory: bit 15 of a hazard code) gather M0's row of the head
    const char* M0c = a.M0 ? static_cast<const char*>(a.M0) + (chain % a.H) * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16
                           : Mc;
    const bool lazy = a.M0 != nullptr;
    // undo log of the backward: the pre-write chunk of every written row, in storage bits
    char* undo_c = a.undo ? static_cast<char*>(a.undo) + dbyte + c * 16 : nullptr;
    const char* vrange = static_cast<const char*>(a.v) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte;
    char* yb = static_cast<char*>(a.y) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    const int T = a.T;
    const int64_t tok0 = chain * T;
    const uint32_t N = static_cast<uint32_t>(a.N);
    // my slots n = g*SPT + j: rows-ring / written-ring offsets of slot j = 0, chunk c
    const uint32_t my_rows = rows0 + (g * SPT * DCH + c) * 16;
    const uint32_t my_wring = wring0 + (g * SPT * DCH + c) * 16;
    const uint32_t wring_c = wring0 + c * 16;
    bool my_w[SPT], my_r[SPT];
#pragma unroll
    for (int j = 0; j < SPT; ++j) { my_w[j] = g * SPT + j < kw; my_r[j] = g * SPT + j < kr; }

    // per-lane pieces of a token's lists (16-byte copies when vec_lists): source base, stride, offset
    const int qw = kw / 4, qr = kr / 4, qm = kmax / 4;
    const int npieces = 2 * qw + 2 * qr + qm;
    const char* psrc[3];
    uint32_t pstride[3], poff[3];
    bool pvalid[3];
#pragma unroll
    for (int q = 0; q < 3; ++q) {
        const int p = lane + 32 * q;
        pvalid[q] = vec_lists && p < npieces;
        const char* src = reinterpret_cast<const char*>(a.idx_w);
        uint32_t stride = kw * 4, off = 0, sub = 0;
        if (p < qw) { src = reinterpret_cast<const char*>(a.idx_w); stride = kw * 4; off = 0; sub = p; }
        else if (p < 2 * qw) { src = reinterpret_cast<const char*>(a.w_w); stride = kw * 4; off = KP * 4; sub = p - qw; }
        else if (p < 2 * qw + qr) { src = reinterpret_cast<const char*>(a.idx_r); stride = kr * 4; off = 2 * KP * 4; sub = p - 2 * qw; }
        else if (p < 2 * qw + 2 * qr) { src = reinterpret_cast<const char*>(a.w_r); stride = kr * 4; off = 3 * KP * 4; sub = p - 2 * qw - qr; }
        else { src = reinterpret_cast<const char*>(hz); stride = kmax * 4; off = 4 * KP * 4; sub = p - 2 * qw - 2 * qr; }
        psrc[q] = src + tok0 * stride + sub * 16;
        pstride[q] = stride;
        poff[q] = off + sub * 16;
    }

    auto copy_meta = [&](int t, uint32_t slot_addr) {
        if (t >= T) return;
        if (vec_lists) {
#pragma unroll
            for (int q = 0; q < 3; ++q)
                if (pvalid[q]) cp_async16z(slot_addr + poff[q], psrc[q] + static_cast<int64_t>(t) * pstride[q], 16);
        } else {
            int* dst = reinterpret_cast<int*>(meta_gen + (slot_addr - meta0));
            const int64_t tok = tok0 + t;
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
        if (lane < DCH) cp_async16z(slot_addr + 5 * KP * 4 + lane * 16, vrange + static_cast<int64_t>(t) * rowbytes + lane * 16, 16);
    };
    // rows that token t gathers (own slots, own chunk), zero-filled for invalid slots
    auto copy_rows = [&](int t, uint32_t meta_addr, uint32_t rows_slot) {
        if (t >= T) return;
        const int* m = reinterpret_cast<const int*>(meta_gen + (meta_addr - meta0));
        int iw[SPT], ir[SPT], hc[SPT];
        lds_vec<SPT>(m + g * SPT, iw);
        lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
        if (lazy) lds_vec<SPT>(m + 4 * KP + g * SPT, hc);
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            if (!lazy) hc[j] = 0;
            const bool ow = my_w[j] && static_cast<uint32_t>(iw[j]) < N;
            const bool orr = my_r[j] && static_cast<uint32_t>(ir[j]) < N;
            const char* bw = (hc[j] & 0x8000) ? M0c : Mc;
            const char* br = hc[j] < 0 ? M0c : Mc;             // bit 31: fresh read slot
            cp_async16z(rows_slot + j * SLOTB, bw + static_cast<uint64_t>(ow ? iw[j] : 0) * rowbytes, ow ? 16 : 0);
            cp_async16z(rows_slot + KS * SLOTB + j * SLOTB, br + static_cast<uint64_t>(orr ? ir[j] : 0) * rowbytes, orr ? 16 : 0);
        }
    };

    // gates: lane i holds token 32 * blk + i; broadcast with a shuffle
    float a_cur = 0.f, b_cur = 0.f, a_nxt = 0.f, b_nxt = 0.f;
    if (lane < T) { a_nxt = load_elem<D>(a.alpha, tok0 + lane); b_nxt = load_elem<D>(a.beta, tok0 + lane); }

    // prologue: lists of tokens [0, LA); then rows of [0, LA) with lists of [LA, 2LA)
    for (int u = 0; u < LA; ++u) copy_meta(u, meta0 + u * meta_stride);
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    for (int u = 0; u < LA; ++u) {
        copy_rows(u, meta0 + u * meta_stride, my_rows + u * 2 * KS * SLOTB);
        copy_meta(u + LA, meta0 + (u + LA) * meta_stride);
        cp_async_commit();
    }

    bool bad = false;
    int ms = 0, rs = 0, ws = 0;                  // ring positions of token t: t % MR, t % LA, t % RING
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
        const uint32_t mslot = meta0 + ms * meta_stride;
        const int* m = reinterpret_cast<const int*>(meta_gen + ms * meta_stride);
        const uint32_t rslot = my_rows + rs * 2 * KS * SLOTB;
        int iw[SPT], ir[SPT], hzv[SPT];
        float ww[SPT], wr[SPT];
        lds_vec<SPT>(m + g * SPT, iw);
        lds_vec<SPT>(m + KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(ww));
        lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
        lds_vec<SPT>(m + 3 * KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(wr));
        lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);

        // ---- gathers (stale rows replaced from the written ring), decay, partial sums.
        // Element math in fp32 pairs on the packed fp32x2 units (each lane of a pair rounds
        // like the scalar operation).
        float2 r[SPT][E2];
        float2 pp[E2], yp[E2];
#pragma unroll
        for (int e = 0; e < E2; ++e) { pp[e] = make_float2(0.f, 0.f); yp[e] = make_float2(0.f, 0.f); }
        const float2 alpha2 = make_float2(alpha, alpha);
        bool fix = false;
        bool okw[SPT];
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            okw[j] = my_w[j] && static_cast<uint32_t>(iw[j]) < N;
            const bool okr = my_r[j] && static_cast<uint32_t>(ir[j]) < N;
            bad |= (my_w[j] && !okw[j]) || (my_r[j] && !okr);
            // hazard codes of unused or invalid slots are garbage: never decode them
            const int hw = okw[j] ? (hzv[j] & 0x7fff) : 0;
            const int hr = okr ? ((hzv[j] >> 16) & 0x7fff) : 0;
            const int dw = (hw - 1) >> 6, dr = (hr - 1) >> 6;
            int rw = ws - dw; rw += rw < 0 ? RING : 0;
            int rr = ws - dr; rr += rr < 0 ? RING : 0;
            const uint32_t aw = hw ? wring_c + (rw * KS + ((hw - 1) & 63)) * SLOTB : rslot + j * SLOTB;
            const bool rfix = hr && dr == 0;             // slot written by this token: added after the write
            const uint32_t ar = (hr && !rfix) ? wring_c + (rr * KS + ((hr - 1) & 63)) * SLOTB : rslot + (KS + j) * SLOTB;
            fix |= rfix && okr;
            const uint4 mw = lds128(aw);
            if (undo_c && okw[j])
                *reinterpret_cast<uint4*>(undo_c + ((tok0 + t) * kw + g * SPT + j) * static_cast<int64_t>(rowbytes)) = mw;
            const uint4 mr = lds128(ar);
            float2 f[E2], h[E2];
            unpack16x2<D>(mw, f);
            unpack16x2<D>(mr, h);
            const float wj = okw[j] ? ww[j] : 0.f;
            const float rho = (okr && !rfix) ? wr[j] : 0.f;
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
        unpack16x2<D>(lds128(mslot + 5 * KP * 4 + c * 16), d2);
#pragma unroll
        for (int e = 0; e < E2; ++e) d2[e] = __fadd2_rn(d2[e], make_float2(-pp[e].x, -pp[e].y));
        const uint32_t wslot = my_wring + ws * KS * SLOTB;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const float bw = beta * ww[j];
            const float2 bw2 = make_float2(bw, bw);
            float2 o[E2];
#pragma unroll
            for (int e = 0; e < E2; ++e) o[e] = __ffma2_rn(bw2, d2[e], r[j][e]);
            const uint4 packed = pack16x2<D>(o);
            if (okw[j]) *reinterpret_cast<uint4*>(Mw + static_cast<uint64_t>(iw[j]) * rowbytes) = packed;
            sts128(wslot + j * SLOTB, packed, okw[j]);
        }
        float delta[E];
#pragma unroll
        for (int e = 0; e < E2; ++e) { delta[2 * e] = d2[e].x; delta[2 * e + 1] = d2[e].y; }
        // ---- reads of slots this token wrote (rare): recompute the writer's value
        if (__any_sync(0xffffffffu, fix)) {
            float yc[E];
#pragma unroll
            for (int e = 0; e < E; ++e) yc[e] = 0.f;
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                const int hr = (hzv[j] >> 16) & 0x7fff;
                const bool okr = my_r[j] && static_cast<uint32_t>(ir[j]) < N;
                if (okr && hr && ((hr - 1) >> 6) == 0) {
                    const int np = (hr - 1) & 63;
                    const int hwn = m[4 * KP + np] & 0x7fff;        // the writer's own hazard code
                    uint32_t ab = rslot + (KS + j) * SLOTB;       // same prefetch as the writer's
                    if (hwn) {
                        int rw = ws - ((hwn - 1) >> 6); rw += rw < 0 ? RING : 0;
                        ab = wring_c + (rw * KS + ((hwn - 1) & 63)) * SLOTB;
                    }
                    float f[E], o[E];
                    unpack16<D>(lds128(ab), f);
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
        if (g == 0) *reinterpret_cast<uint4*>(yb + static_cast<int64_t>(t) * rowbytes) = pack16x2<D>(yp);
        // ---- prefetch: rows of token t+LA (rows slot of token t), lists of token t+2LA (slot of t-1)
        {
            int mfut = ms + LA; mfut -= mfut >= MR ? MR : 0;
            copy_rows(t + LA, meta0 + mfut * meta_stride, rslot);
            int mnew = ms + 2 * LA; mnew -= mnew >= MR ? MR : 0;
            copy_meta(t + 2 * LA, meta0 + mnew * meta_stride);
            cp_async_commit();
        }
        ms = ms + 1 == MR ? 0 : ms + 1;
        rs = rs + 1 == LA ? 0 : rs + 1;
        ws = ws + 1 == RING ? 0 : ws + 1;
    }
    cp_async_wait<0>();
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
}

template <class D, int DCH, int SPT, int LA>
cudaError_t launch_rec_kernel(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    const int wpc = p.wpc > 0 ? p.wpc : 1;
    const size_t smem = wpc * rec_warp_smem_bytes(LA, (32 / DCH) * SPT, DCH);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur<D, DCH, SPT, LA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t warps = static_cast<int64_t>(a.B) * a.H * p.nsplit;
    k_recur<D, DCH, SPT, LA><<<static_cast<unsigned>((warps + wpc - 1) / wpc), 32 * wpc, smem, s>>>(a, p.nsplit, hz,
                                                                                                 p.kmax, vec_lists);
    return cudaGetLastError();
}

template <class D, int DCH, int SPT, int LA>
cudaError_t launch_rec_split(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s);

template <class D, int DCH, int SPT>
cudaError_t launch_rec_la(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vl, cudaStream_t s) {
    if (p.la == 1) return launch_rec_kernel<D, DCH, SPT, 1>(p, a, hz, vl, s);
    return p.split ? launch_rec_split<D, DCH, SPT, 4>(p, a, hz, vl, s) : launch_rec_kernel<D, DCH, SPT, 4>(p, a, hz, vl, s);
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

namespace sdm {

// ------------------------------------------------------------------------------------------
// K-REC, writer/reader split.  One CTA of two warps per (chain, d-range): warp 0 does the
// decay, prediction and delta write of token t (Eqs. sdm-decay, sdm-write) while warp 1
// does the read of token t-1 (Eq. sdm-read), so each warp's per-token instruction chain is
// about half of the fused one.  They meet in the ring of rows written by the last LA+1
// tokens (read-gathers of slots written in the hazard window, including by the token itself,
// take the writer's row from there) and hand over through two mbarriers:
//   written[t] (writer -> reader): token t's rows are in memory and in the ring;
//   read[t]    (reader -> writer): token t is read, so ring entry t - LA is free again.
// The writer of token t waits for read[t-1] only before its stores; the reader of token t
// waits for written[t].  Neither can run two phases ahead of the other, so the waits on
// phase parity are unambiguous.  Every wait is bounded; on timeout both warps leave the
// token loop and the device status gets its timeout bit.
// ------------------------------------------------------------------------------------------
constexpr long long REC_WAIT_CYCLES = 4000000000LL;    // ~2 s at 2 GHz

__host__ __device__ inline size_t rec_split_smem_bytes(int la, int ks, int dch) {
    return static_cast<size_t>(2) * la * ks * dch * 16                // prefetched rows: write, read
         + static_cast<size_t>(la + 1) * ks * dch * 16                // rows written lately
         + static_cast<size_t>(2) * (2 * la + 1) * rec_meta_stride(ks, dch)   // lists, per warp
         + 32;                                                        // two mbarriers + abort flag
}

__device__ __forceinline__ void rec_mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
// Bounded wait for the completion of the phase with parity `par`; false on timeout or abort.
__device__ __forceinline__ bool rec_mbar_wait(uint32_t bar, uint32_t par, volatile int* abort_flag, long long limit) {
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(ok) : "r"(bar), "r"(par) : "memory");
        if (ok) return true;
        if (*abort_flag || clock64() - t0 > limit) return false;
    }
}

template <class D, int DCH, int SPT, int LA>
__global__ void __launch_bounds__(64) k_recur_split(const RecArgs a, int nsplit, const int32_t* __restrict__ hz,
                                                    int kmax, int vec_lists) {
    static_assert(LA >= 1, "look-ahead");
    constexpr int E = D::E;
    constexpr int E2 = E / 2;
    constexpr int G = 32 / DCH;
    constexpr int KS = G * SPT;
    constexpr int KP = rec_ks_pad(KS);
    constexpr int MR = 2 * LA + 1;
    constexpr int RING = LA + 1;
    constexpr uint32_t SLOTB = DCH * 16;
    extern __shared__ __align__(16) unsigned char smS[];
    const int warp = threadIdx.x >> 5;                       // 0: writer, 1: reader
    const int lane = threadIdx.x & 31;
    const int meta_stride = static_cast<int>(rec_meta_stride(KS, DCH));
    const uint32_t sm0 = static_cast<uint32_t>(__cvta_generic_to_shared(smS));
    const uint32_t rows0 = sm0 + warp * (LA * KS * SLOTB);                   // own [LA][KS][DCH] x 16 B
    const uint32_t wring0 = sm0 + 2 * LA * KS * SLOTB;                      // shared [RING][KS][DCH] x 16 B
    const uint32_t metab = wring0 + RING * KS * SLOTB;
    const uint32_t meta0 = metab + warp * MR * meta_stride;                 // own [MR][stride]
    unsigned char* meta_gen = smS + (meta0 - sm0);
    const uint32_t bar_written = metab + 2 * MR * meta_stride;
    const uint32_t bar_read = bar_written + 8;
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smS + (bar_written - sm0) + 16);
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(bar_written) : "memory");
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(bar_read) : "memory");
        *abort_flag = 0;
    }
    __syncthreads();

    const int c = lane % DCH;
    const int g = lane / DCH;
    const int kw = a.kw, kr = a.kr;
    const int kmine = warp == 0 ? kw : kr;                   // list this warp gathers
    const int64_t chain = blockIdx.x / nsplit;
    const int split = blockIdx.x - static_cast<int>(chain) * nsplit;
    const uint32_t rowbytes = static_cast<uint32_t>(a.dv) * D::BYTES;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;
    const char* Mc = static_cast<const char*>(a.mem) + chain * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    char* Mw = const_cast<char*>(Mc);
    // fresh slots (lazy initial memory: bit 15 of a hazard code) gather M0's row of the head
    const char* M0c = a.M0 ? static_cast<const char*>(a.M0) + (chain % a.H) * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16
                           : Mc;
    const bool lazy = a.M0 != nullptr;
    // undo log of the backward: the pre-write chunk of every written row, in storage bits
    char* undo_c = a.undo ? static_cast<char*>(a.undo) + dbyte + c * 16 : nullptr;
    const char* vrange = static_cast<const char*>(a.v) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte;
    char* yb = static_cast<char*>(a.y) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    const int T = a.T;
    const int64_t tok0 = chain * T;
    const uint32_t N = static_cast<uint32_t>(a.N);
    const uint32_t my_rows = rows0 + (g * SPT * DCH + c) * 16;
    const uint32_t my_wring = wring0 + (g * SPT * DCH + c) * 16;
    const uint32_t wring_c = wring0 + c * 16;
    bool mine[SPT];
#pragma unroll
    for (int j = 0; j < SPT; ++j) mine[j] = g * SPT + j < kmine;

    // lists of token t (16-byte pieces when vec_lists; same layout as the fused kernel)
    const int qw = kw / 4, qr = kr / 4;
    const int npieces = 2 * qw + 2 * qr + kmax / 4;
    const char* psrc[3];
    uint32_t pstride[3], poff[3];
    bool pvalid[3];
#pragma unroll
    for (int q = 0; q < 3; ++q) {
        const int p = lane + 32 * q;
        pvalid[q] = vec_lists && p < npieces;
        const char* src = reinterpret_cast<const char*>(a.idx_w);
        uint32_t stride = kw * 4, off = 0, sub = 0;
        if (p < qw) { src = reinterpret_cast<const char*>(a.idx_w); stride = kw * 4; off = 0; sub = p; }
        else if (p < 2 * qw) { src = reinterpret_cast<const char*>(a.w_w); stride = kw * 4; off = KP * 4; sub = p - qw; }
        else if (p < 2 * qw + qr) { src = reinterpret_cast<const char*>(a.idx_r); stride = kr * 4; off = 2 * KP * 4; sub = p - 2 * qw; }
        else if (p < 2 * qw + 2 * qr) { src = reinterpret_cast<const char*>(a.w_r); stride = kr * 4; off = 3 * KP * 4; sub = p - 2 * qw - qr; }
        else { src = reinterpret_cast<const char*>(hz); stride = kmax * 4; off = 4 * KP * 4; sub = p - 2 * qw - 2 * qr; }
        psrc[q] = src + tok0 * stride + sub * 16;
        pstride[q] = stride;
        poff[q] = off + sub * 16;
    }
    auto copy_meta = [&](int t, uint32_t slot_addr) {
        if (t >= T) return;
        if (vec_lists) {
#pragma unroll
            for (int q = 0; q < 3; ++q)
                if (pvalid[q]) cp_async16z(slot_addr + poff[q], psrc[q] + static_cast<int64_t>(t) * pstride[q], 16);
        } else {
            int* dst = reinterpret_cast<int*>(meta_gen + (slot_addr - meta0));
            const int64_t tok = tok0 + t;
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
        if (warp == 0 && lane < DCH)
            cp_async16z(slot_addr + 5 * KP * 4 + lane * 16, vrange + static_cast<int64_t>(t) * rowbytes + lane * 16, 16);
    };
    // rows token t gathers from this warp's list (writer: write slots; reader: read slots)
    const int list_off = warp == 0 ? 0 : 2 * KP;
    auto copy_rows = [&](int t, uint32_t meta_addr, uint32_t rows_slot) {
        if (t >= T) return;
        const int* m = reinterpret_cast<const int*>(meta_gen + (meta_addr - meta0));
        int ix[SPT], hc[SPT];
        lds_vec<SPT>(m + list_off + g * SPT, ix);
        if (lazy) lds_vec<SPT>(m + 4 * KP + g * SPT, hc);
#pragma unroll
        for (int j = 0; j < SPT; ++j)
            if (!lazy) hc[j] = 0;
        const int fresh_bit = warp == 0 ? 0x8000 : static_cast<int>(0x80000000u);   // write / read half
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const bool ok = mine[j] && static_cast<uint32_t>(ix[j]) < N;
            const char* src = (hc[j] & fresh_bit) ? M0c : Mc;
            cp_async16z(rows_slot + j * SLOTB, src + static_cast<uint64_t>(ok ? ix[j] : 0) * rowbytes, ok ? 16 : 0);
        }
    };

    // prologue: lists of tokens [0, LA); then rows of [0, LA) with lists of [LA, 2LA)
    for (int u = 0; u < LA; ++u) copy_meta(u, meta0 + u * meta_stride);
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    for (int u = 0; u < LA; ++u) {
        copy_rows(u, meta0 + u * meta_stride, my_rows + u * KS * SLOTB);
        copy_meta(u + LA, meta0 + (u + LA) * meta_stride);
        cp_async_commit();
    }
    auto prefetch = [&](int t, int ms, int rs) {     // rows of t+LA into the slot of t; lists of t+2LA
        int mfut = ms + LA; mfut -= mfut >= MR ? MR : 0;
        copy_rows(t + LA, meta0 + mfut * meta_stride, my_rows + rs * KS * SLOTB);
        int mnew = ms + 2 * LA; mnew -= mnew >= MR ? MR : 0;
        copy_meta(t + 2 * LA, meta0 + mnew * meta_stride);
        cp_async_commit();
    };

    bool bad = false, timed_out = false;
    const long long wait_limit = a.wait_cycles > 0 ? a.wait_cycles : REC_WAIT_CYCLES;
    if (warp == 0) {
        // ------------------------------------------------------------------ writer
        float a_cur = 0.f, b_cur = 0.f, a_nxt = 0.f, b_nxt = 0.f;
        if (lane < T) { a_nxt = load_elem<D>(a.alpha, tok0 + lane); b_nxt = load_elem<D>(a.beta, tok0 + lane); }
        int ms = 0, rs = 0, ws = 0;
        for (int t = 0; t < T; ++t) {
            if ((t & 31) == 0) {
                a_cur = a_nxt; b_cur = b_nxt;
                const int tn = t + 32 + lane;
                if (tn < T) { a_nxt = load_elem<D>(a.alpha, tok0 + tn); b_nxt = load_elem<D>(a.beta, tok0 + tn); }
            }
            const float alpha = __shfl_sync(0xffffffffu, a_cur, t & 31);
            const float beta = __shfl_sync(0xffffffffu, b_cur, t & 31);
            cp_async_wait<LA - 1>();
            __syncwarp();
            const int* m = reinterpret_cast<const int*>(meta_gen + ms * meta_stride);
            const uint32_t rslot = my_rows + rs * KS * SLOTB;
            int iw[SPT], hzv[SPT];
            float ww[SPT];
            lds_vec<SPT>(m + g * SPT, iw);
            lds_vec<SPT>(m + KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(ww));
            lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);
            float2 r[SPT][E2];
            float2 pp[E2];
#pragma unroll
            for (int e = 0; e < E2; ++e) pp[e] = make_float2(0.f, 0.f);
            const float2 alpha2 = make_float2(alpha, alpha);
            bool okw[SPT];
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                okw[j] = mine[j] && static_cast<uint32_t>(iw[j]) < N;
                bad |= mine[j] && !okw[j];
                const int hw = okw[j] ? (hzv[j] & 0x7fff) : 0;      // never decode unused slots
                int rw = ws - ((hw - 1) >> 6); rw += rw < 0 ? RING : 0;
                const uint32_t aw = hw ? wring_c + (rw * KS + ((hw - 1) & 63)) * SLOTB : rslot + j * SLOTB;
                float2 f[E2];
                const uint4 mw = lds128(aw);
                if (undo_c && okw[j])
                    *reinterpret_cast<uint4*>(undo_c + ((tok0 + t) * kw + g * SPT + j) * static_cast<int64_t>(rowbytes)) = mw;
                unpack16x2<D>(mw, f);
                const float wj = okw[j] ? ww[j] : 0.f;
                const float2 wj2 = make_float2(wj, wj);
#pragma unroll
                for (int e = 0; e < E2; ++e) {
                    r[j][e] = __fmul2_rn(alpha2, f[e]);
                    pp[e] = __ffma2_rn(wj2, r[j][e], pp[e]);
                }
            }
#pragma unroll
            for (int off = DCH; off < 32; off <<= 1) {
#pragma unroll
                for (int e = 0; e < E2; ++e)
                    pp[e] = __fadd2_rn(pp[e], make_float2(__shfl_xor_sync(0xffffffffu, pp[e].x, off),
                                                          __shfl_xor_sync(0xffffffffu, pp[e].y, off)));
            }
            float2 d2[E2];
            unpack16x2<D>(lds128(meta0 + ms * meta_stride + 5 * KP * 4 + c * 16), d2);
#pragma unroll
            for (int e = 0; e < E2; ++e) d2[e] = __fadd2_rn(d2[e], make_float2(-pp[e].x, -pp[e].y));
            uint4 packed[SPT];
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                const float bw = beta * ww[j];
                const float2 bw2 = make_float2(bw, bw);
                float2 o[E2];
#pragma unroll
                for (int e = 0; e < E2; ++e) o[e] = __ffma2_rn(bw2, d2[e], r[j][e]);
                packed[j] = pack16x2<D>(o);
            }
            // ring entry of token t - LA - 1 is free once the reader is done with token t - 1
            if (t > 0 && !rec_mbar_wait(bar_read, static_cast<uint32_t>((t - 1) & 1), abort_flag, wait_limit)) {
                timed_out = true;
                break;
            }
            const uint32_t wslot = my_wring + ws * KS * SLOTB;
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                if (okw[j]) *reinterpret_cast<uint4*>(Mw + static_cast<uint64_t>(iw[j]) * rowbytes) = packed[j];
                sts128(wslot + j * SLOTB, packed[j], okw[j]);
            }
            __syncwarp();
            if (lane == 0 && !(a.hold_handover && t == 0)) rec_mbar_arrive(bar_written);
            prefetch(t, ms, rs);
            ms = ms + 1 == MR ? 0 : ms + 1;
            rs = rs + 1 == LA ? 0 : rs + 1;
            ws = ws + 1 == RING ? 0 : ws + 1;
        }
    } else {
        // ------------------------------------------------------------------ reader
        int ms = 0, rs = 0, ws = 0;
        for (int t = 0; t < T; ++t) {
            cp_async_wait<LA - 1>();
            __syncwarp();
            const int* m = reinterpret_cast<const int*>(meta_gen + ms * meta_stride);
            const uint32_t rslot = my_rows + rs * KS * SLOTB;
            int ir[SPT], hzv[SPT];
            float wr[SPT];
            lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
            lds_vec<SPT>(m + 3 * KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(wr));
            lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);
            if (!rec_mbar_wait(bar_written, static_cast<uint32_t>(t & 1), abort_flag, wait_limit)) {
                timed_out = true;
                break;
            }
            float2 yp[E2];
#pragma unroll
            for (int e = 0; e < E2; ++e) yp[e] = make_float2(0.f, 0.f);
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                const bool okr = mine[j] && static_cast<uint32_t>(ir[j]) < N;
                bad |= mine[j] && !okr;
                const int hr = okr ? ((hzv[j] >> 16) & 0x7fff) : 0;
                int rr = ws - ((hr - 1) >> 6); rr += rr < 0 ? RING : 0;
                const uint32_t ar = hr ? wring_c + (rr * KS + ((hr - 1) & 63)) * SLOTB : rslot + j * SLOTB;
                float2 h[E2];
                unpack16x2<D>(lds128(ar), h);
                const float rho = okr ? wr[j] : 0.f;
                const float2 rho2 = make_float2(rho, rho);
#pragma unroll
                for (int e = 0; e < E2; ++e) yp[e] = __ffma2_rn(rho2, h[e], yp[e]);
            }
            __syncwarp();
            if (lane == 0) rec_mbar_arrive(bar_read);          // ring reads of token t done
#pragma unroll
            for (int off = DCH; off < 32; off <<= 1) {
#pragma unroll
                for (int e = 0; e < E2; ++e)
                    yp[e] = __fadd2_rn(yp[e], make_float2(__shfl_xor_sync(0xffffffffu, yp[e].x, off),
                                                          __shfl_xor_sync(0xffffffffu, yp[e].y, off)));
            }
            if (g == 0) *reinterpret_cast<uint4*>(yb + static_cast<int64_t>(t) * rowbytes) = pack16x2<D>(yp);
            prefetch(t, ms, rs);
            ms = ms + 1 == MR ? 0 : ms + 1;
            rs = rs + 1 == LA ? 0 : rs + 1;
            ws = ws + 1 == RING ? 0 : ws + 1;
        }
    }
    if (timed_out) *abort_flag = 1;
    cp_async_wait<0>();
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, timed_out) && lane == 0) flag_error(a.err, ERR_TIMEOUT);
}

template <class D, int DCH, int SPT, int LA>
cudaError_t launch_rec_split(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    const size_t smem = rec_split_smem_bytes(LA, (32 / DCH) * SPT, DCH);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur_split<D, DCH, SPT, LA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    k_recur_split<D, DCH, SPT, LA><<<static_cast<unsigned>(chains * p.nsplit), 64, smem, s>>>(a, p.nsplit, hz, p.kmax,
                                                                                                vec_lists);
    return cudaGetLastError();
}

}  // namespace sdm
