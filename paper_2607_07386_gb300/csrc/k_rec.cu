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
// Latency hiding.  The addressing does not depend on the memory, so the gathers of token
// t+LA (both the write-gather and the read-gather) are issued while token t is processed,
// into a register ring; slot lists and weights are loaded 2*LA tokens ahead.  A prefetched
// row is stale if a token in between wrote that slot: the hazard pass (k_hazard) records,
// for every (t, n), the most recent writer (t - delta, n') within the window (delta in
// [1, LA-1] for the write-gather, [0, LA-1] for the read-gather, delta = 0 being the
// read-after-write of the token itself).  Every written row is also kept in a shared
// ring of the last LA tokens, from which hazarded values are taken.  Ordering: each
// token's scatter is made visible by a block barrier before any later gather is issued.
#include "sdm_internal.h"

namespace sdm {

// ------------------------------------------------------------------------------------------
// Hazard pass.  hz[(chain*T + t)*kmax + n] = write code (low 16 bits) | read code << 16;
// code 0 = no hazard, else 1 + delta*64 + n' (writer t - delta, position n' of its list).
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
        if (n < a.kw && LA > 1) {
            const int s = __ldg(iw + n);
            for (int d = 1; d < LA && d <= t; ++d) {
                const int p = find_sorted(a.idx_w + (tok - d) * a.kw, a.kw, s);
                if (p >= 0) { cw = 1 + d * 64 + p; break; }
            }
        }
        if (n < a.kr) {
            const int s = __ldg(ir + n);
            for (int d = 0; d < LA && d <= t; ++d) {
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
template <class D, int DCH, int SPT, int LA>
__global__ void __launch_bounds__(512) k_recur(const RecArgs a, int nsplit, const int32_t* __restrict__ hz, int kmax) {
    constexpr int E = D::E;
    constexpr int MR = 2 * LA;                      // depth of the slot-list ring
    extern __shared__ __align__(16) float smR[];
    const int nthreads = blockDim.x;
    const int NW = nthreads >> 5;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c = tid % DCH;
    const int g = tid / DCH;
    const int G = nthreads / DCH;
    float* red0 = smR;                                          // [NW][DCH][E] prediction partials
    float* red1 = smR + NW * DCH * E;                           // [NW][DCH][E] read partials
    uint4* wring = reinterpret_cast<uint4*>(smR + 2 * NW * DCH * E);   // [LA][kw][DCH] rows written lately

    const int64_t chain = blockIdx.x / nsplit;
    const int split = blockIdx.x - static_cast<int>(chain) * nsplit;
    const int64_t rowbytes = static_cast<int64_t>(a.dv) * D::BYTES;
    const int64_t coff = static_cast<int64_t>(split * DCH + c) * 16;
    char* Mb = static_cast<char*>(a.mem) + chain * a.N * rowbytes + coff;
    const char* vb = static_cast<const char*>(a.v) + chain * a.T * rowbytes + coff;
    char* yb = static_cast<char*>(a.y) + chain * a.T * rowbytes + coff;
    const int T = a.T;

    // slot-list ring (registers): written slot, weight, read slot, weight, hazard codes
    int m_iw[MR][SPT], m_ir[MR][SPT], m_hz[MR][SPT];
    float m_ww[MR][SPT], m_wr[MR][SPT];
    // gather ring (registers): write-gather and read-gather chunks, v chunk, gates
    uint4 g_w[LA][SPT], g_r[LA][SPT], g_v[LA];
    float g_al[LA], g_be[LA];

    auto load_meta = [&](int t, int slot) {
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
            int iw = -1, ir = -1, h = 0;
            float ww = 0.f, wr = 0.f;
            if (t < T) {
                const int64_t tok = chain * T + t;
                if (n < a.kw) {
                    iw = __ldg(a.idx_w + tok * a.kw + n);
                    ww = __ldg(a.w_w + tok * a.kw + n);
                    if (iw < 0 || iw >= a.N) { flag_error(a.err, ERR_BAD_INDEX); iw = -1; }
                }
                if (n < a.kr) {
                    ir = __ldg(a.idx_r + tok * a.kr + n);
                    wr = __ldg(a.w_r + tok * a.kr + n);
                    if (ir < 0 || ir >= a.N) { flag_error(a.err, ERR_BAD_INDEX); ir = -1; }
                }
                if (n < kmax) h = __ldg(hz + tok * kmax + n);
            }
            m_iw[slot][j] = iw; m_ww[slot][j] = ww; m_ir[slot][j] = ir; m_wr[slot][j] = wr; m_hz[slot][j] = h;
        }
    };
    auto issue_gather = [&](int t, int ms, int gs) {
        if (t >= T) return;
        const int64_t tok = chain * T + t;
        g_al[gs] = load_elem<D>(a.alpha, tok);
        g_be[gs] = load_elem<D>(a.beta, tok);
        g_v[gs] = *reinterpret_cast<const uint4*>(vb + t * rowbytes);
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int iw = m_iw[ms][j], ir = m_ir[ms][j];
            g_w[gs][j] = iw >= 0 ? *reinterpret_cast<const uint4*>(Mb + iw * rowbytes) : make_uint4(0, 0, 0, 0);
            g_r[gs][j] = ir >= 0 ? *reinterpret_cast<const uint4*>(Mb + ir * rowbytes) : make_uint4(0, 0, 0, 0);
        }
    };
    auto consume = [&](int t, int ms, int gs) {
        const float alpha = g_al[gs], beta = g_be[gs];
        float r[SPT][E];
        float part[E];
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            uint4 m = g_w[gs][j];
            const int h = m_hz[ms][j] & 0xffff;
            if (h) {   // slot written after the prefetch: take the row from the ring
                const int d = (h - 1) >> 6, np = (h - 1) & 63;
                m = wring[(((t - d) % LA) * a.kw + np) * DCH + c];
            }
            float f[E];
            unpack16<D>(m, f);
#pragma unroll
            for (int e = 0; e < E; ++e) {
                r[j][e] = alpha * f[e];
                part[e] = fmaf(m_ww[ms][j], r[j][e], part[e]);
            }
        }
#pragma unroll
        for (int e = 0; e < E; ++e)
            for (int off = DCH; off < 32; off <<= 1) part[e] += __shfl_xor_sync(0xffffffffu, part[e], off);
        if (lane < DCH) {
#pragma unroll
            for (int e = 0; e < E; ++e) red0[(warp * DCH + c) * E + e] = part[e];
        }
        __syncthreads();                                            // B1: prediction partials
        float dv[E];
        unpack16<D>(g_v[gs], dv);
        for (int w = 0; w < NW; ++w) {
#pragma unroll
            for (int e = 0; e < E; ++e) dv[e] -= red0[(w * DCH + c) * E + e];
        }
        // delta = v - v~ (the subtraction of the partials in warp order equals v - sum)
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            const int n = g + j * G;
            const int iw = m_iw[ms][j];
            if (iw >= 0) {
                const float bw = beta * m_ww[ms][j];
                float o[E];
#pragma unroll
                for (int e = 0; e < E; ++e) o[e] = fmaf(bw, dv[e], r[j][e]);
                const uint4 packed = pack16<D>(o);
                *reinterpret_cast<uint4*>(Mb + iw * rowbytes) = packed;
                wring[(((t % LA) * a.kw) + n) * DCH + c] = packed;
            }
        }
        __syncthreads();                                            // B2: scatter and ring visible
#pragma unroll
        for (int e = 0; e < E; ++e) part[e] = 0.f;
#pragma unroll
        for (int j = 0; j < SPT; ++j) {
            uint4 m = g_r[gs][j];
            const int h = (m_hz[ms][j] >> 16) & 0xffff;
            if (h) {
                const int d = (h - 1) >> 6, np = (h - 1) & 63;
                m = wring[(((t - d) % LA) * a.kw + np) * DCH + c];
            }
            float f[E];
            unpack16<D>(m, f);
#pragma unroll
            for (int e = 0; e < E; ++e) part[e] = fmaf(m_wr[ms][j], f[e], part[e]);
        }
#pragma unroll
        for (int e = 0; e < E; ++e)
            for (int off = DCH; off < 32; off <<= 1) part[e] += __shfl_xor_sync(0xffffffffu, part[e], off);
        if (lane < DCH) {
#pragma unroll
            for (int e = 0; e < E; ++e) red1[(warp * DCH + c) * E + e] = part[e];
        }
        __syncthreads();                                            // B3: read partials
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
    };

    // prologue: lists of tokens [0, 2LA), gathers of tokens [0, LA)
#pragma unroll
    for (int u = 0; u < MR; ++u) load_meta(u, u);
#pragma unroll
    for (int u = 0; u < LA; ++u) issue_gather(u, u, u);

    for (int t0 = 0; t0 < T; t0 += MR) {
#pragma unroll
        for (int u = 0; u < MR; ++u) {
            const int t = t0 + u;
            if (t >= T) break;
            consume(t, u, u % LA);
            issue_gather(t + LA, (u + LA) % MR, u % LA);
            load_meta(t + MR, u);
        }
    }
}

template <class D, int DCH, int SPT, int LA>
static cudaError_t launch_rec_typed(const RecArgs& a, int nsplit, int threads, const int32_t* hz, int kmax,
                                    cudaStream_t stream) {
    const size_t sm = static_cast<size_t>(2) * (threads / 32) * DCH * D::E * sizeof(float) +
                      static_cast<size_t>(LA) * a.kw * DCH * 16;
    if (sm > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_recur<D, DCH, SPT, LA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(sm));
        if (e != cudaSuccess) return e;
    }
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    k_recur<D, DCH, SPT, LA><<<static_cast<unsigned>(chains * nsplit), threads, sm, stream>>>(a, nsplit, hz, kmax);
    return cudaGetLastError();
}

RecPlan rec_plan(int dtype, int B, int H, int T, int dv, int kw, int kr) {
    RecPlan p{};
    const int bytes = dtype == 0 ? 4 : 2;
    const int nch = dv * bytes / 16;                       // 16-byte chunks per row
    const int64_t chains = static_cast<int64_t>(B) * H;
    int dch = 1;
    while (dch < 32 && nch % (dch * 2) == 0) dch *= 2;    // largest power-of-two divisor <= 32
    // finest d-split (>= one 32-byte sector per row) that still leaves few CTAs per SM
    while (dch > 2 && chains * (nch / dch) < 512) dch /= 2;
    p.dch = dch;
    p.nsplit = nch / dch;
    const int kmax = kw > kr ? kw : kr;
    p.kmax = kmax;
    // slot groups: about one slot per thread, at most 512 threads
    int threads = ((kmax * dch + 31) / 32) * 32;
    if (threads > 512) threads = 512;
    if (threads < 32) threads = 32;
    int spt = (kmax + threads / dch - 1) / (threads / dch);
    p.spt = spt <= 1 ? 1 : spt <= 2 ? 2 : 4;   // threads * 4 >= kmax * dch holds for kmax <= 64, dch <= 32
    p.threads = threads;
    p.la = T <= 1 ? 1 : (p.spt <= 1 ? 4 : p.spt <= 2 ? 2 : 1);
    return p;
}

template <class D, int DCH>
static cudaError_t launch_dch(const RecPlan& p, const RecArgs& a, const int32_t* hz, cudaStream_t s) {
    const int key = p.spt * 16 + p.la;
    switch (key) {
        case 1 * 16 + 1: return launch_rec_typed<D, DCH, 1, 1>(a, p.nsplit, p.threads, hz, p.kmax, s);
        case 1 * 16 + 4: return launch_rec_typed<D, DCH, 1, 4>(a, p.nsplit, p.threads, hz, p.kmax, s);
        case 2 * 16 + 1: return launch_rec_typed<D, DCH, 2, 1>(a, p.nsplit, p.threads, hz, p.kmax, s);
        case 2 * 16 + 2: return launch_rec_typed<D, DCH, 2, 2>(a, p.nsplit, p.threads, hz, p.kmax, s);
        case 4 * 16 + 1: return launch_rec_typed<D, DCH, 4, 1>(a, p.nsplit, p.threads, hz, p.kmax, s);
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
        case 32: return launch_dch<D, 32>(p, a, hz, s);
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
