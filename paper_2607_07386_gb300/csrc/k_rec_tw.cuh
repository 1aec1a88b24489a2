// K-REC, token-interleaved form: several warps advance one (chain, d-range) together, warp w
// taking the tokens t = w (mod W).  Each warp runs the fused token body of k_recur (decay,
// prediction, delta write, read of the post-write memory; Eqs. sdm-decay, sdm-write,
// sdm-read) on its own tokens, so W tokens of a chain are in flight at once and the chain is
// no longer bound by the latency of one token's instruction chain.
//
// Order between the warps.  Tokens only depend on each other through memory rows.  Each warp
// publishes two progress words in shared memory, each after a block-scope fence: the last
// of its tokens whose gathers have landed, and the last whose stores are done.
//   * read after write: a warp issues the row prefetch of its token t' only once every token
//     before t' - LA is done (LA = (P + 1) W), so a prefetched row can only be stale if a token
//     in [t' - LA, t' - 1] wrote the slot; the hazard pass marks exactly those gathers.  For a
//     marked gather the warp waits until the writer token is done and reloads the row from
//     memory (L2): rare, a few per thousand gathers at N = 2^18.  A read of a slot the same
//     token writes recomputes the written value from the same operands, bit for bit;
//   * write after write: a token that writes a slot an earlier token of the window wrote has
//     a write-gather hazard on it, so it waits for that writer before it writes;
//   * write after read: when a token of the window read-gathers a slot that token t writes,
//     t stores its rows only once every token up to that reader has gathered (the warps'
//     gather words), so no earlier gather sees a later write.  Readers older than the window
//     were done before t's rows were prefetched.
// Every wait is bounded: on timeout the CTA sets the timeout bit and leaves.
#pragma once
#include "sdm_internal.h"

namespace sdm {

__host__ __device__ inline size_t tw_warp_smem_bytes(int p, int ks, int dch) {
    const size_t b = static_cast<size_t>(p) * 2 * ks * dch * 16                 // prefetched rows
                   + static_cast<size_t>(2 * p + 1) * rec_meta_stride(ks, dch);  // lists, v
    return (b + 127) / 128 * 128;
}
__host__ __device__ inline size_t tw_smem_bytes(int w, int p, int ks, int dch) {
    return static_cast<size_t>(w) * tw_warp_smem_bytes(p, ks, dch) + 256;       // + progress words
}

__device__ __forceinline__ uint4 ldcg16(const void* p) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];\n" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

// Bounded wait until progress word prog[ww] reaches `u`; false on timeout or abort.
__device__ __forceinline__ bool tw_wait_done(volatile int* prog, int ww, int u, volatile int* abort_flag, long long limit) {
    if (prog[ww] >= u) return true;
    const long long t0 = clock64();
    while (prog[ww] < u) {
        if (*abort_flag || clock64() - t0 > limit) return false;
        __nanosleep(64);                 // leave the issue slots to the warps doing work
    }
    return true;
}

template <class D, int DCH, int SPT, int W, int P>
__global__ void __launch_bounds__(32 * W) k_recur_tw(const RecArgs a, int nsplit, const int32_t* __restrict__ hz,
                                                     int kmax, int vec_lists) {
    constexpr int E = D::E;
    constexpr int E2 = E / 2;
    constexpr int G = 32 / DCH;
    constexpr int KS = G * SPT;
    constexpr int KP = rec_ks_pad(KS);
    constexpr int MR = 2 * P + 1;
    constexpr int LA = (P + 1) * W;                       // hazard window (tokens)
    constexpr uint32_t SLOTB = DCH * 16;
    extern __shared__ __align__(128) unsigned char smT[];
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    const uint32_t smbase = static_cast<uint32_t>(__cvta_generic_to_shared(smT));
    const uint32_t wbytes = static_cast<uint32_t>(tw_warp_smem_bytes(P, KS, DCH));
    const uint32_t rows0 = smbase + w * wbytes;                               // [P][2][KS][DCH] x 16 B
    const uint32_t meta0 = rows0 + P * 2 * KS * SLOTB;                        // [MR][stride]
    unsigned char* meta_gen = smT + (meta0 - smbase);
    const int meta_stride = static_cast<int>(rec_meta_stride(KS, DCH));
    // progress words: prog[v] = last token of warp v whose stores are done, gath[v] = last
    // token whose gathers have landed (both start at the "token before the first")
    volatile int* prog = reinterpret_cast<volatile int*>(smT + W * wbytes);
    volatile int* gath = prog + 16;
    volatile int* abort_flag = prog + 32;
    if (threadIdx.x < W) {
        prog[threadIdx.x] = static_cast<int>(threadIdx.x) - W;
        gath[threadIdx.x] = static_cast<int>(threadIdx.x) - W;
    }
    if (threadIdx.x == 0) *abort_flag = 0;
    __syncthreads();

    const long long limit = a.wait_cycles > 0 ? a.wait_cycles : 4000000000LL;
    const int c = lane % DCH;
    const int g = lane / DCH;
    const int kw = a.kw, kr = a.kr;
    const int64_t chain = blockIdx.x / nsplit;
    const int split = static_cast<int>(blockIdx.x - chain * nsplit);
    const uint32_t rowbytes = static_cast<uint32_t>(a.dv) * D::BYTES;
    const bool row256 = rowbytes % 256 == 0;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;
    const char* Mc = static_cast<const char*>(a.mem) + chain * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    char* Mw = const_cast<char*>(Mc);
    const char* M0c = a.M0 ? static_cast<const char*>(a.M0) + (chain % a.H) * a.N * static_cast<int64_t>(rowbytes) + dbyte + c * 16
                           : Mc;
    const bool lazy = a.M0 != nullptr;
    char* undo_c = a.undo ? static_cast<char*>(a.undo) + dbyte + c * 16 : nullptr;
    const char* vrange = static_cast<const char*>(a.v) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte;
    char* yb = static_cast<char*>(a.y) + chain * a.T * static_cast<int64_t>(rowbytes) + dbyte + c * 16;
    const int T = a.T;
    const int64_t tok0 = chain * T;
    const uint32_t N = static_cast<uint32_t>(a.N);
    bool my_w[SPT], my_r[SPT];
#pragma unroll
    for (int j = 0; j < SPT; ++j) { my_w[j] = g * SPT + j < kw; my_r[j] = g * SPT + j < kr; }

    // per-lane 16-byte pieces of a token's lists (as in k_recur)
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
    // rows that token t gathers (own slots, own chunk) into rows slot `rows_t`; zero-filled for
    // invalid slots; fresh slots of the lazy memory come from M0.  Each 16-byte piece asks L2 to
    // fetch the whole aligned 256-byte region around it (the row, at d_v = 128 bf16), so DRAM
    // moves rows as whole bursts and the other d-ranges' pieces of a row hit L2 (random 64-byte
    // pieces alone reach less than half of the bandwidth of whole 256-byte rows).
    auto copy_rows = [&](int t, uint32_t meta_addr, uint32_t rows_t) {
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
            const char* bw = (hc[j] & HZ_W_FRESH) ? M0c : Mc;
            const char* br = (hc[j] & HZ_R_FRESH) ? M0c : Mc;
            const uint32_t at = rows_t + ((g * SPT + j) * DCH + c) * 16;
            cp_async16z_row(at, bw + static_cast<uint64_t>(ow ? iw[j] : 0) * rowbytes, ow ? 16 : 0, row256);
            cp_async16z_row(at + KS * SLOTB, br + static_cast<uint64_t>(orr ? ir[j] : 0) * rowbytes, orr ? 16 : 0, row256);
        }
    };
    // own tokens: t = w + i * W, i = 0, 1, ...
    const int nown = T > w ? (T - w + W - 1) / W : 0;
    auto tok_of = [&](int i) { return w + i * W; };

    // gates: lane l holds own token 32 * blk + l
    float a_cur = 0.f, b_cur = 0.f, a_nxt = 0.f, b_nxt = 0.f;
    if (lane < nown) { a_nxt = load_elem<D>(a.alpha, tok0 + tok_of(lane)); b_nxt = load_elem<D>(a.beta, tok0 + tok_of(lane)); }

    // prologue: lists of own tokens [0, P); then rows of [0, P) with lists of [P, 2P).  Tokens
    // before w + (P - 1) W < LA need no progress check.
    for (int u = 0; u < P; ++u) copy_meta(u < nown ? tok_of(u) : T, meta0 + u * meta_stride);
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    for (int u = 0; u < P; ++u) {
        copy_rows(u < nown ? tok_of(u) : T, meta0 + u * meta_stride, rows0 + u * 2 * KS * SLOTB);
        copy_meta(u + P < nown ? tok_of(u + P) : T, meta0 + (u + P) * meta_stride);
        cp_async_commit();
    }

    bool bad = false, timed_out = false;
    int ms = 0, rs = 0;
    for (int i = 0; i < nown; ++i) {
        const int t = tok_of(i);
        if ((i & 31) == 0) {
            a_cur = a_nxt; b_cur = b_nxt;
            const int in = i + 32 + lane;
            if (in < nown) { a_nxt = load_elem<D>(a.alpha, tok0 + tok_of(in)); b_nxt = load_elem<D>(a.beta, tok0 + tok_of(in)); }
        }
        const float alpha = __shfl_sync(0xffffffffu, a_cur, i & 31);
        const float beta = __shfl_sync(0xffffffffu, b_cur, i & 31);
        cp_async_wait<P - 1>();         // own rows of token t and lists of own token i + P have landed
        __syncwarp();
        const uint32_t mslot = meta0 + ms * meta_stride;
        const int* m = reinterpret_cast<const int*>(meta_gen + ms * meta_stride);
        const uint32_t rows_t = rows0 + rs * 2 * KS * SLOTB;
        const uint32_t my_rows = rows_t + (g * SPT * DCH + c) * 16;
        int iw[SPT], ir[SPT], hzv[SPT];
        float ww[SPT], wr[SPT];
        lds_vec<SPT>(m + g * SPT, iw);
        lds_vec<SPT>(m + KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(ww));
        lds_vec<SPT>(m + 2 * KP + g * SPT, ir);
        lds_vec<SPT>(m + 3 * KP + g * SPT, *reinterpret_cast<int(*)[SPT]>(wr));
        lds_vec<SPT>(m + 4 * KP + g * SPT, hzv);

        // ---- stale prefetches (rare): wait for the writer token, reload the row from memory
        bool okw[SPT], okr[SPT], stale = false, fix = false;
        int war_u = -1;                                  // latest earlier reader of a write slot
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            okw[j] = my_w[j] && static_cast<uint32_t>(iw[j]) < N;
            okr[j] = my_r[j] && static_cast<uint32_t>(ir[j]) < N;
            bad |= (my_w[j] && !okw[j]) || (my_r[j] && !okr[j]);
            const int hw = okw[j] ? hz_wcode(hzv[j]) : 0;
            const int hr = okr[j] ? hz_rcode(hzv[j]) : 0;
            stale |= hw != 0 || hr > 64;                 // read codes 1..64: written by this token
            fix |= hr != 0 && hr <= 64;
            const int war = okw[j] ? hz_war(hzv[j]) : 0;
            war_u = war ? max(war_u, t - war) : war_u;
        }
        if (__any_sync(0xffffffffu, stale)) {
#pragma unroll
            for (int j = 0; j < SPT; ++j) {
                const int hw = okw[j] ? hz_wcode(hzv[j]) : 0;
                const int hr = okr[j] ? hz_rcode(hzv[j]) : 0;
                if (hw != 0) {
                    const int u = t - ((hw - 1) >> 6);
                    if (!tw_wait_done(prog, u % W, u, abort_flag, limit)) timed_out = true;
                    __threadfence_block();
                    sts128(my_rows + j * SLOTB, ldcg16(Mw + static_cast<uint64_t>(iw[j]) * rowbytes), true);
                }
                if (hr > 64) {
                    const int u = t - ((hr - 1) >> 6);
                    if (!tw_wait_done(prog, u % W, u, abort_flag, limit)) timed_out = true;
                    __threadfence_block();
                    sts128(my_rows + (KS + j) * SLOTB, ldcg16(Mw + static_cast<uint64_t>(ir[j]) * rowbytes), true);
                }
            }
            if (__any_sync(0xffffffffu, timed_out)) break;
        }
        // ---- publish: token t's gathers have landed (in shared memory)
        __syncwarp();
        if (lane == 0 && !(a.hold_handover && t == 0)) {     // (test hook: withheld for token 0)
            __threadfence_block();
            gath[w] = t;
        }

        // ---- gathers, decay, partial sums (packed fp32x2 math, as in k_recur)
        float2 r[SPT][E2];
        float2 pp[E2], yp[E2];
#pragma unroll
        for (int e = 0; e < E2; ++e) { pp[e] = make_float2(0.f, 0.f); yp[e] = make_float2(0.f, 0.f); }
        const float2 alpha2 = make_float2(alpha, alpha);
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int hr = okr[j] ? hz_rcode(hzv[j]) : 0;
            const bool rfix = hr != 0 && hr <= 64;
            const uint4 mw = lds128(my_rows + j * SLOTB);
            if (undo_c && okw[j])
                *reinterpret_cast<uint4*>(undo_c + ((tok0 + t) * kw + g * SPT + j) * static_cast<int64_t>(rowbytes)) = mw;
            const uint4 mr = lds128(my_rows + (KS + j) * SLOTB);
            float2 f[E2], h[E2];
            unpack16x2<D>(mw, f);
            unpack16x2<D>(mr, h);
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
        // ---- delta = v - v~ and the write, once every earlier token has gathered
        float2 d2[E2];
        unpack16x2<D>(lds128(mslot + 5 * KP * 4 + c * 16), d2);
#pragma unroll
        for (int e = 0; e < E2; ++e) d2[e] = __fadd2_rn(d2[e], make_float2(-pp[e].x, -pp[e].y));
        if (a.hold_handover && t > 0) war_u = max(war_u, 0);   // (test hook: every later token waits)
        war_u = __reduce_max_sync(0xffffffffu, war_u);
        if (war_u >= 0) {                                // (rare) every token up to that reader gathered
            bool ok = true;
#pragma unroll
            for (int v = 0; v < W; ++v) ok &= tw_wait_done(gath, v, war_u - W + 1, abort_flag, limit);
            if (!ok) timed_out = true;
            if (__any_sync(0xffffffffu, timed_out)) break;
            __threadfence_block();
        }
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const float bw = beta * ww[j];
            const float2 bw2 = make_float2(bw, bw);
            float2 o[E2];
#pragma unroll
            for (int e = 0; e < E2; ++e) o[e] = __ffma2_rn(bw2, d2[e], r[j][e]);
            if (okw[j]) *reinterpret_cast<uint4*>(Mw + static_cast<uint64_t>(iw[j]) * rowbytes) = pack16x2<D>(o);
        }
        // ---- reads of slots this token wrote (rare): recompute the writer's value from the
        // writer's gathered row (the write half of this token's rows, at the writer's position)
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
                if (hr != 0 && hr <= 64) {
                    const int np = hr - 1;
                    float f[E], o[E];
                    unpack16<D>(lds128(rows_t + (np * DCH + c) * 16), f);
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
        // ---- publish: token t's stores are done
        __syncwarp();
        if (lane == 0) {
            __threadfence_block();
            prog[w] = t;
        }
        // ---- prefetch own token i + P (rows, once every token before it - LA is done) into
        // the rows slot of token t; lists of own token i + 2P into the slot of own token i - 1
        {
            const int tp = i + P < nown ? tok_of(i + P) : T;
            if (tp < T) {
                const int need = tp - LA - W;                  // every warp done with a token >= need
                bool ok = true;
#pragma unroll
                for (int v = 0; v < W; ++v) ok &= tw_wait_done(prog, v, need, abort_flag, limit);
                if (!ok) timed_out = true;
                if (__any_sync(0xffffffffu, timed_out)) break;
                __threadfence_block();
            }
            int mfut = ms + P; mfut -= mfut >= MR ? MR : 0;
            copy_rows(tp, meta0 + mfut * meta_stride, rows_t);
            int mnew = ms + 2 * P; mnew -= mnew >= MR ? MR : 0;
            copy_meta(i + 2 * P < nown ? tok_of(i + 2 * P) : T, meta0 + mnew * meta_stride);
            cp_async_commit();
        }
        ms = ms + 1 == MR ? 0 : ms + 1;
        rs = rs + 1 == P ? 0 : rs + 1;
    }
    if (timed_out) *abort_flag = 1;
    cp_async_wait<0>();
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (__any_sync(0xffffffffu, timed_out) && lane == 0) flag_error(a.err, ERR_TIMEOUT);
}

template <class D, int DCH, int SPT, int W, int P>
cudaError_t launch_rec_tw(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s) {
    const size_t smem = tw_smem_bytes(W, P, (32 / DCH) * SPT, DCH);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur_tw<D, DCH, SPT, W, P>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t ctas = static_cast<int64_t>(a.B) * a.H * p.nsplit;
    k_recur_tw<D, DCH, SPT, W, P><<<static_cast<unsigned>(ctas), 32 * W, smem, s>>>(a, p.nsplit, hz, p.kmax, vec_lists);
    return cudaGetLastError();
}

}  // namespace sdm
