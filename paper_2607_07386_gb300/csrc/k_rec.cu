// K-REC: fused sparse gated delta recurrence (Eqs. sdm-decay, sdm-write, sdm-read).
//
// For one (b, h) chain, tokens in order t = 0 .. T-1:
//   r_n  = alpha_t * M[I^w_t[n]]                 (decay of the written slots only)
//   v~   = sum_n w_n r_n                         (prediction)
//   M[I^w_t[n]] = R(r_n + beta_t w_n (v_t - v~)) (delta write, storage rounding R)
//   y_t  = R(sum_n rho_n M[I^r_t[n]])            (read of the post-write memory)
//
// Layout of the work.  Every step is elementwise along d_v once (idx, w) are fixed, so a
// chain is split into independent d-ranges: one CTA owns one (chain, d-range) and thread
// (g, c) moves 16-byte chunk c of the rows of slot group g (slots n = g, g+G, ...), i.e.
// rows are read and written as coalesced 16-byte vectors.  The prediction and the read are
// reduced over slot groups with warp shuffles and one shared-memory pass.
//
// Latency hiding.  The addressing does not depend on the memory, so the rows token t+LA
// will gather (write-gather and read-gather) are copied into a shared-memory ring with
// cp.async while token t is processed; slot lists, weights, hazard codes and v are copied
// 2*LA tokens ahead.  A prefetched row is stale if a token in between wrote that slot: the
// hazard pass (k_hazard) records, for every (t, n), the most recent writer (t - delta, n')
// with delta in [1, LA] for the write-gather and [0, LA] for the read-gather (delta = 0:
// the token reads a slot it has just written).  Every written row is kept in a shared ring
// of the last LA+1 tokens, from which stale rows are replaced; a delta = 0 read recomputes
// the written value from the same operands as the writer (bit-identical), so one block
// barrier per token suffices.  A prefetch issued at token t may miss token t's own stores,
// which is why the window reaches delta = LA.
#include "sdm_internal.h"

namespace sdm {

// ------------------------------------------------------------------------------------------
// Hazard pass.  hz[(chain*T + t)*kmax + n] = write code (low 16 bits) | read code << 16;
// code 0 = no hazard, else 1 + delta*64 + n' (writer t - delta, position n' of its list),
// delta in [1, LA] for the write-gather and [0, LA] for the read-gather.
// Slot lists must be ascending within each token (as the addressing produces them).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ int find_sorted(const int32_t* list, int k, int s) {
    int lo = 0, hi = k - 1;
    while (lo <= hi) {
        const int mid = (lo + hi) >> 1;
        const int v = __ldg(list + mid);
        if (v == s) return mid;
        if (v < s) lo = mid + 1; else hi = mid - 1;
    }
    return -1;
}

__global__ void __launch_bounds__(256) k_hazard(const RecArgs a, int LA, int kmax, int32_t* hz) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.H * a.T;
    const int64_t tok = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
    if (tok >= BT) return;
    const int64_t chain = tok / a.T;
    const int t = static_cast<int>(tok - chain * a.T);
    const int32_t* iw = a.idx_w + tok * a.kw;
    const int32_t* ir = a.idx_r + tok * a.kr;
    bool sorted = true;
    for (int n = 1; n < a.kw; ++n) sorted &= __ldg(iw + n - 1) < __ldg(iw + n);
    for (int n = 1; n < a.kr; ++n) sorted &= __ldg(ir + n - 1) < __ldg(ir + n);
    if (!sorted) flag_error(a.err, ERR_UNSORTED);
    for (int n = 0; n < kmax; ++n) {
        int cw = 0, cr = 0;
        if (n < a.kw) {
            const int s = __ldg(iw + n);
            for (int d = 1; d <= LA && d <= t; ++d) {
                const int p = find_sorted(a.idx_w + (tok - d) * a.kw, a.kw, s);
                if (p >= 0) { cw = 1 + d * 64 + p; break; }
            }
        }
        if (n < a.kr) {
            const int s = __ldg(ir + n);
            for (int d = 0; d <= LA && d <= t; ++d) {
                const int p = find_sorted(a.idx_w + (tok - d) * a.kw, a.kw, s);
                if (p >= 0) { cr = 1 + d * 64 + p; break; }
            }
        }
        hz[tok * kmax + n] = cw | (cr << 16);
    }
}

// ------------------------------------------------------------------------------------------
// Recurrence
// ------------------------------------------------------------------------------------------
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

// Shared-memory layout of one recurrence CTA (see rec_smem_bytes).
struct RecSmem {
    int KS;          // slot capacity per token: G * SPT
    int meta_words;  // 32-bit words of one token's lists: 2 kw + 2 kr + kmax
    size_t rows, wring, meta, red0, red1, total;
};

__host__ __device__ inline RecSmem rec_smem(int la, int KS, int kw, int kr, int kmax, int dch, int nw, int E) {
    RecSmem m{};
    m.KS = KS;
    m.meta_words = 2 * kw + 2 * kr + kmax;
    size_t off = 0;
    m.rows = off;  off += static_cast<size_t>(la) * 2 * KS * dch * 16;                 // prefetched rows
    m.wring = off; off += static_cast<size_t>(la + 1) * kw * dch * 16;                 // rows written lately
    m.meta = off;  off += static_cast<size_t>(2 * la + 1) * (((m.meta_words * 4 + 15) / 16) * 16 + dch * 16);
    m.red0 = off;  off += static_cast<size_t>(2) * nw * dch * E * 4;
    m.red1 = off;  off += static_cast<size_t>(2) * nw * dch * E * 4;
    m.total = off;
    return m;
}

template <class D, int DCH, int SPT, int LA>
__global__ void __launch_bounds__(256) k_recur(const RecArgs a, int nsplit, const int32_t* __restrict__ hz, int kmax) {
    constexpr int E = D::E;
    constexpr int MR = 2 * LA + 1;                 // token lists in flight (ring depth)
    extern __shared__ __align__(16) unsigned char smR[];
    const int nthreads = blockDim.x;
    const int NW = nthreads >> 5;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c = tid % DCH;                       // 16-byte chunk within the CTA's d-range
    const int g = tid / DCH;                       // slot group
    const int G = nthreads / DCH;
    const int kw = a.kw, kr = a.kr;
    const RecSmem L = rec_smem(LA, G * SPT, kw, kr, kmax, DCH, NW, E);
    uint4* rows = reinterpret_cast<uint4*>(smR + L.rows);       // [LA][2][KS][DCH]
    uint4* wring = reinterpret_cast<uint4*>(smR + L.wring);     // [LA+1][kw][DCH]
    unsigned char* meta = smR + L.meta;                          // [MR][lists | v chunks]
    float* red0 = reinterpret_cast<float*>(smR + L.red0);       // [2][NW][DCH][E]
    float* red1 = reinterpret_cast<float*>(smR + L.red1);       // [2][NW][DCH][E]
    const int meta_lists = ((L.meta_words * 4 + 15) / 16) * 16;
    const int meta_stride = meta_lists + DCH * 16;
    const int KS = L.KS;

    const int64_t chain = blockIdx.x / nsplit;
    const int split = blockIdx.x - static_cast<int>(chain) * nsplit;
    const int64_t rowbytes = static_cast<int64_t>(a.dv) * D::BYTES;
    const int64_t dbyte = static_cast<int64_t>(split * DCH) * 16;   // first byte of the CTA's d-range
    char* Mb = static_cast<char*>(a.mem) + chain * a.N * rowbytes + dbyte + c * 16;
    const char* vrange = static_cast<const char*>(a.v) + chain * a.T * rowbytes + dbyte;
    char* yb = static_cast<char*>(a.y) + chain * a.T * rowbytes + dbyte + c * 16;
    const int T = a.T;
    const int64_t tok0 = chain * T;

    // token lists of token t -> meta slot t % MR: iw[kw] ww[kw] ir[kr] wr[kr] hz[kmax] | v[DCH]
    auto m_iw = [&](int slot) { return reinterpret_cast<int*>(meta + slot * meta_stride); };
    auto m_ww = [&](int slot) { return reinterpret_cast<float*>(meta + slot * meta_stride) + kw; };
    auto m_ir = [&](int slot) { return reinterpret_cast<int*>(meta + slot * meta_stride) + 2 * kw; };
    auto m_wr = [&](int slot) { return reinterpret_cast<float*>(meta + slot * meta_stride) + 2 * kw + kr; };
    auto m_hz = [&](int slot) { return reinterpret_cast<int*>(meta + slot * meta_stride) + 2 * kw + 2 * kr; };
    auto m_v = [&](int slot) { return reinterpret_cast<uint4*>(meta + slot * meta_stride + meta_lists); };

    auto copy_meta = [&](int t) {
        if (t >= T) return;
        const int slot = t % MR;
        const int64_t tok = tok0 + t;
        unsigned char* dst = meta + slot * meta_stride;
        for (int p = tid; p < L.meta_words; p += nthreads) {
            const void* src;
            if (p < kw) src = a.idx_w + tok * kw + p;
            else if (p < 2 * kw) src = a.w_w + tok * kw + (p - kw);
            else if (p < 2 * kw + kr) src = a.idx_r + tok * kr + (p - 2 * kw);
            else if (p < 2 * kw + 2 * kr) src = a.w_r + tok * kr + (p - 2 * kw - kr);
            else src = hz + tok * kmax + (p - 2 * kw - 2 * kr);
            cp_async4(dst + p * 4, src);
        }
        if (tid < DCH) cp_async16(dst + meta_lists + tid * 16, vrange + t * rowbytes + tid * 16);
    };
    // rows token t will gather (own slots, own chunk) -> rows slot t % LA
    auto copy_rows = [&](int t) {
        if (t >= T) return;
        const int slot = t % LA, ms = t % MR;
        const int* iw = m_iw(ms);
        const int* ir = m_ir(ms);
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
            if (n < kw) {
                const int s = iw[n];
                if (s >= 0 && s < a.N) cp_async16(&rows[((slot * 2 + 0) * KS + n) * DCH + c], Mb + s * rowbytes);
            }
            if (n < kr) {
                const int s = ir[n];
                if (s >= 0 && s < a.N) cp_async16(&rows[((slot * 2 + 1) * KS + n) * DCH + c], Mb + s * rowbytes);
            }
        }
    };
    auto block_sync = [&]() {
        if (NW > 1) __syncthreads(); else __syncwarp();
    };

    // gates: lane i of every warp holds token (32 * blk + i); broadcast with a shuffle
    float a_cur = 0.f, b_cur = 0.f, a_nxt = 0.f, b_nxt = 0.f;
    if (lane < T) { a_nxt = load_elem<D>(a.alpha, tok0 + lane); b_nxt = load_elem<D>(a.beta, tok0 + lane); }

    // prologue: lists of tokens [0, LA), then rows of [0, LA) with lists of [LA, 2LA)
    for (int u = 0; u < LA; ++u) copy_meta(u);
    cp_async_commit();
    cp_async_wait<0>();
    block_sync();
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
        cp_async_wait<LA - 1>();                 // own rows of token t and lists of token t+LA landed
        const int ms = t % MR, rs = t % LA, ws = t % (LA + 1);
        const int* iw = m_iw(ms);
        const float* ww = m_ww(ms);
        const int* ir = m_ir(ms);
        const float* wr = m_wr(ms);
        const int* hzt = m_hz(ms);
        // ---- write-gather (stale rows from the ring), decay, partial prediction
        float r[SPT][E];
        float part[E];
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
#pragma unroll
            for (int e = 0; e < E; ++e) r[j][e] = 0.f;
            if (n < kw) {
                const int s = iw[n];
                if (s >= 0 && s < a.N) {
                    const int h = hzt[n] & 0xffff;
                    uint4 m;
                    if (h) {
                        const int d = (h - 1) >> 6, np = (h - 1) & 63;
                        m = wring[(((t - d) % (LA + 1)) * kw + np) * DCH + c];
                    } else {
                        m = rows[((rs * 2 + 0) * KS + n) * DCH + c];
                    }
                    float f[E];
                    unpack16<D>(m, f);
                    const float w = ww[n];
#pragma unroll
                    for (int e = 0; e < E; ++e) {
                        r[j][e] = alpha * f[e];
                        part[e] = fmaf(w, r[j][e], part[e]);
                    }
                } else {
                    flag_error(a.err, ERR_BAD_INDEX);
                }
            }
        }
#pragma unroll
        for (int e = 0; e < E; ++e)
            for (int off = DCH; off < 32; off <<= 1) part[e] += __shfl_xor_sync(0xffffffffu, part[e], off);
        float pred[E];
        if (NW > 1) {
            if (lane < DCH) {
#pragma unroll
                for (int e = 0; e < E; ++e) red0[(((t & 1) * NW + warp) * DCH + c) * E + e] = part[e];
            }
        }
        block_sync();                             // the one barrier of token t
        if (NW > 1) {
            if (t > 0 && g == 0) {                // y of the previous token (read partials)
                float yv[E];
#pragma unroll
                for (int e = 0; e < E; ++e) yv[e] = 0.f;
                for (int w = 0; w < NW; ++w) {
#pragma unroll
                    for (int e = 0; e < E; ++e) yv[e] += red1[((((t - 1) & 1) * NW + w) * DCH + c) * E + e];
                }
                *reinterpret_cast<uint4*>(yb + (t - 1) * rowbytes) = pack16<D>(yv);
            }
#pragma unroll
            for (int e = 0; e < E; ++e) pred[e] = 0.f;
            for (int w = 0; w < NW; ++w) {
#pragma unroll
                for (int e = 0; e < E; ++e) pred[e] += red0[(((t & 1) * NW + w) * DCH + c) * E + e];
            }
        } else {
#pragma unroll
            for (int e = 0; e < E; ++e) pred[e] = part[e];
        }
        float delta[E];
        unpack16<D>(m_v(ms)[c], delta);
#pragma unroll
        for (int e = 0; e < E; ++e) delta[e] -= pred[e];          // v - v~
        // ---- delta write (scatter + ring)
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
            if (n < kw) {
                const int s = iw[n];
                if (s >= 0 && s < a.N) {
                    const float bw = beta * ww[n];
                    float o[E];
#pragma unroll
                    for (int e = 0; e < E; ++e) o[e] = fmaf(bw, delta[e], r[j][e]);
                    const uint4 packed = pack16<D>(o);
                    *reinterpret_cast<uint4*>(Mb + s * rowbytes) = packed;
                    wring[((ws * kw) + n) * DCH + c] = packed;
                }
            }
        }
        // ---- read of the post-write memory
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
            if (n < kr) {
                const int s = ir[n];
                if (s >= 0 && s < a.N) {
                    const int h = (hzt[n] >> 16) & 0xffff;
                    uint4 m = rows[((rs * 2 + 1) * KS + n) * DCH + c];
                    if (h) {
                        const int d = (h - 1) >> 6, np = (h - 1) & 63;
                        if (d > 0) {
                            m = wring[(((t - d) % (LA + 1)) * kw + np) * DCH + c];
                        } else {
                            // slot written by this token at position np: recompute the writer's value
                            const int hw = hzt[np] & 0xffff;
                            uint4 base = m;   // the pre-write row (same prefetch as the writer's)
                            if (hw) {
                                const int d2 = (hw - 1) >> 6, np2 = (hw - 1) & 63;
                                base = wring[(((t - d2) % (LA + 1)) * kw + np2) * DCH + c];
                            }
                            float f[E], o[E];
                            unpack16<D>(base, f);
                            const float bw = beta * ww[np];
#pragma unroll
                            for (int e = 0; e < E; ++e) o[e] = fmaf(bw, delta[e], alpha * f[e]);
                            m = pack16<D>(o);
                        }
                    }
                    float f[E];
                    unpack16<D>(m, f);
                    const float rho = wr[n];
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
        if (NW > 1) {
            if (lane < DCH) {
#pragma unroll
                for (int e = 0; e < E; ++e) red1[(((t & 1) * NW + warp) * DCH + c) * E + e] = part[e];
            }
        } else if (g == 0) {
            *reinterpret_cast<uint4*>(yb + t * rowbytes) = pack16<D>(part);
        }
        // ---- prefetch: rows of token t+LA, lists of token t+2LA (slot of token t-1)
        copy_rows(t + LA);
        copy_meta(t + 2 * LA);
        cp_async_commit();
    }
    if (NW > 1) {
        __syncthreads();
        if (T > 0 && g == 0) {
            float yv[E];
#pragma unroll
            for (int e = 0; e < E; ++e) yv[e] = 0.f;
            for (int w = 0; w < NW; ++w) {
#pragma unroll
                for (int e = 0; e < E; ++e) yv[e] += red1[((((T - 1) & 1) * NW + w) * DCH + c) * E + e];
            }
            *reinterpret_cast<uint4*>(yb + (T - 1) * rowbytes) = pack16<D>(yv);
        }
    }
    cp_async_wait<0>();
}

RecPlan rec_plan(int dtype, int B, int H, int T, int dv, int kw, int kr) {
    RecPlan p{};
    const int bytes = dtype == 0 ? 4 : 2;
    const int E = 16 / bytes;
    const int nch = dv * bytes / 16;                       // 16-byte chunks per row
    const int64_t chains = static_cast<int64_t>(B) * H;
    const int kmax = kw > kr ? kw : kr;
    p.kmax = kmax;
    int dch = 1;
    while (dch < 16 && nch % (dch * 2) == 0) dch *= 2;    // whole row per CTA when possible (<= 256 B)
    // split rows across CTAs (keeping >= 64-byte pieces) until there are enough CTAs
    while (dch * 16 > 64 && chains * (nch / dch) < 128) dch /= 2;
    p.dch = dch;
    p.nsplit = nch / dch;
    // about 4 slots per thread; at least one warp; at most 256 threads
    int G = (kmax + 3) / 4;
    if (G * dch < 32) G = 32 / dch;
    while (G * dch > 256) G /= 2;
    int threads = G * dch;
    threads = (threads + 31) / 32 * 32;
    G = threads / dch;
    p.threads = threads;
    const int spt = (kmax + G - 1) / G;
    p.spt = spt <= 1 ? 1 : spt <= 2 ? 2 : spt <= 4 ? 4 : 8;
    // lookahead: the deepest ring that fits the shared memory the CTAs of one SM can share
    const int64_t ctas = chains * p.nsplit;
    const int per_sm = static_cast<int>((ctas + 147) / 148);
    const size_t budget = (per_sm <= 1 ? 200u : 200u / static_cast<unsigned>(per_sm)) * 1024u;
    p.la = 1;
    if (T > 1) {
        for (int la = 8; la >= 2; la /= 2) {
            if (rec_smem(la, G * p.spt, kw, kr, kmax, dch, threads / 32, E).total <= budget) { p.la = la; break; }
        }
    }
    p.smem = rec_smem(p.la, G * p.spt, kw, kr, kmax, dch, threads / 32, E).total;
    return p;
}

template <class D, int DCH, int SPT, int LA>
static cudaError_t launch_rec_typed(const RecPlan& p, const RecArgs& a, const int32_t* hz, cudaStream_t stream) {
    if (p.smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur<D, DCH, SPT, LA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(p.smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    k_recur<D, DCH, SPT, LA><<<static_cast<unsigned>(chains * p.nsplit), p.threads, p.smem, stream>>>(a, p.nsplit, hz,
                                                                                                          p.kmax);
    return cudaGetLastError();
}

template <class D, int DCH, int SPT>
static cudaError_t launch_spt(const RecPlan& p, const RecArgs& a, const int32_t* hz, cudaStream_t s) {
    switch (p.la) {
        case 1: return launch_rec_typed<D, DCH, SPT, 1>(p, a, hz, s);
        case 2: return launch_rec_typed<D, DCH, SPT, 2>(p, a, hz, s);
        case 4: return launch_rec_typed<D, DCH, SPT, 4>(p, a, hz, s);
        case 8: return launch_rec_typed<D, DCH, SPT, 8>(p, a, hz, s);
        default: return cudaErrorInvalidValue;
    }
}

template <class D, int DCH>
static cudaError_t launch_dch(const RecPlan& p, const RecArgs& a, const int32_t* hz, cudaStream_t s) {
    switch (p.spt) {
        case 1: return launch_spt<D, DCH, 1>(p, a, hz, s);
        case 2: return launch_spt<D, DCH, 2>(p, a, hz, s);
        case 4: return launch_spt<D, DCH, 4>(p, a, hz, s);
        case 8: return launch_spt<D, DCH, 8>(p, a, hz, s);
        default: return cudaErrorInvalidValue;
    }
}

template <class D>
static cudaError_t launch_dtype(const RecPlan& p, const RecArgs& a, const int32_t* hz, cudaStream_t s) {
    switch (p.dch) {
        case 1: return launch_dch<D, 1>(p, a, hz, s);
        case 2: return launch_dch<D, 2>(p, a, hz, s);
        case 4: return launch_dch<D, 4>(p, a, hz, s);
        case 8: return launch_dch<D, 8>(p, a, hz, s);
        case 16: return launch_dch<D, 16>(p, a, hz, s);
        default: return cudaErrorInvalidValue;
    }
}

size_t rec_workspace_bytes(int B, int H, int T, int kw, int kr) {
    const int kmax = kw > kr ? kw : kr;
    return static_cast<size_t>(B) * H * T * kmax * sizeof(int32_t);
}

cudaError_t launch_recur(int dtype, const RecArgs& a, int32_t* hz_ws, cudaStream_t stream) {
    const RecPlan p = rec_plan(dtype, a.B, a.H, a.T, a.dv, a.kw, a.kr);
    const int64_t BT = static_cast<int64_t>(a.B) * a.H * a.T;
    k_hazard<<<static_cast<unsigned>((BT + 255) / 256), 256, 0, stream>>>(a, p.la, p.kmax, hz_ws);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return dtype == 0 ? launch_dtype<F32>(p, a, hz_ws, stream) : launch_dtype<BF16>(p, a, hz_ws, stream);
}

}  // namespace sdm
