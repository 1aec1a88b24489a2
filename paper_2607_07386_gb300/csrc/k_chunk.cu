// Chunkwise (WY) form of the recurrence (App. A.1 "Intra-Chunk Parallel vs. Chunkwise
// Recurrent", A.2 "Sparse Inner Product via Two-Pointer Merge").
//
// One CTA per (b, h) chain walks its chunks of C <= 32 tokens in order.  Per chunk, in shared
// memory (fp32):
//   S0  the chunk's slot lists, weights, log(alpha), beta and v;
//   S1  segmented cumulative log-decays: lam_w[t][n] = sum of log(alpha_t') over the chunk's
//       tokens t' <= t that write slot idx_w[t][n] (binary search in their sorted lists), and
//       lam_r[t][n] the same for read slot idx_r[t][n];
//   S2  A[t][s] (s < t, write-write) and QK[t][s] (s <= t, read-write) gated sparse inner
//       products by a two-pointer merge of the sorted lists;
//   S3  forward substitution with the unit lower-triangular M_sys = I + diag(beta) A:
//       dV = M_sys^-1 diag(beta) V and B = M_sys^-1 diag(-beta);
//   S4  retrieved[t] = sum_n w e^lam_w M[idx_w] and inter[t] = sum_n rho e^lam_r M[idx_r],
//       gathered from the chunk-initial memory in HBM;
//   S5  u = dV + B retrieved, y = inter + QK u (y stored, rounded);
//   S6  the last occurrence of each written slot in the chunk (one warp) forms the new row
//       e^lam M[i] + sum over the slot's occurrences of e^(lam - lam_t) w_t u_t, rounded.
// The memory is rounded at chunk boundaries only, like the chunkwise oracle.  First version:
// plain loads and block barriers only; no asynchronous copies, no waits.
#include "sdm_internal.h"

namespace sdm {

constexpr int CK_THREADS = 256;
constexpr int CK_MAXC = 32;

template <class D> __device__ __forceinline__ void store_val(void* base, int64_t i, float v);
template <> __device__ __forceinline__ void store_val<F32>(void* base, int64_t i, float v) {
    reinterpret_cast<float*>(base)[i] = v;
}
template <> __device__ __forceinline__ void store_val<BF16>(void* base, int64_t i, float v) {
    reinterpret_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(v);
}

// position of slot s in the ascending list l[0..k), or -1
__device__ __forceinline__ int find_slot(const int* l, int k, int s) {
    int lo = 0, hi = k;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (l[mid] < s) lo = mid + 1;
        else hi = mid;
    }
    return (lo < k && l[lo] == s) ? lo : -1;
}

__device__ __forceinline__ float gated_ip(const int* ia, const float* va, const float* la, int ka, const int* ib,
                                          const float* vb, const float* lb, int kb) {
    float acc = 0.f;
    int a = 0, b = 0;
    while (a < ka && b < kb) {
        const int x = ia[a], y = ib[b];
        if (x == y) {
            acc = fmaf(va[a] * vb[b], __expf(la[a] - lb[b]), acc);
            ++a;
            ++b;
        } else if (x < y) {
            ++a;
        } else {
            ++b;
        }
    }
    return acc;
}

size_t chunk_smem_bytes(int C, int kw, int kr, int dv) {
    return static_cast<size_t>(4) * (2 * C * kw + 2 * C * kr)      // lists and weights
         + static_cast<size_t>(4) * (C * kw + C * kr)               // lam_w, lam_r
         + static_cast<size_t>(4) * 3 * C                           // log alpha, alpha, beta
         + static_cast<size_t>(4) * 3 * C * C                       // A, QK, B
         + static_cast<size_t>(4) * 3 * C * dv;                     // dV, R (then u), I
}

template <class D>
__global__ void __launch_bounds__(CK_THREADS) k_recur_chunk(const RecArgs a, int C) {
    extern __shared__ __align__(16) unsigned char smC[];
    const int kw = a.kw, kr = a.kr, dv = a.dv, T = a.T;
    const uint32_t N = static_cast<uint32_t>(a.N);
    int* s_iw = reinterpret_cast<int*>(smC);
    float* s_ww = reinterpret_cast<float*>(s_iw + C * kw);
    int* s_ir = reinterpret_cast<int*>(s_ww + C * kw);
    float* s_wr = reinterpret_cast<float*>(s_ir + C * kr);
    float* s_lw = s_wr + C * kr;
    float* s_lr = s_lw + C * kw;
    float* s_la = s_lr + C * kr;
    float* s_al = s_la + C;
    float* s_be = s_al + C;
    float* s_A = s_be + C;
    float* s_QK = s_A + C * C;
    float* s_B = s_QK + C * C;
    float* s_dV = s_B + C * C;
    float* s_R = s_dV + C * dv;
    float* s_I = s_R + C * dv;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t chain = blockIdx.x;
    const int64_t mrow0 = chain * a.N;                       // first memory row of the chain
    bool bad = false, unsorted = false;
    for (int c0 = 0; c0 < T; c0 += C) {
        const int n = min(C, T - c0);
        const int64_t tok0 = chain * T + c0;
        // ---- S0: lists, weights, gates, v
        for (int e = tid; e < n * kw; e += CK_THREADS) {
            const int s = __ldg(a.idx_w + tok0 * kw + e);
            const bool ok = static_cast<uint32_t>(s) < N;
            bad |= !ok;
            // the two-pointer merges and binary searches need strictly ascending lists
            unsorted |= (e % kw) > 0 && __ldg(a.idx_w + tok0 * kw + e - 1) >= s;
            s_iw[e] = s;
            s_ww[e] = ok ? __ldg(a.w_w + tok0 * kw + e) : 0.f;
        }
        for (int e = tid; e < n * kr; e += CK_THREADS) {
            const int s = __ldg(a.idx_r + tok0 * kr + e);
            const bool ok = static_cast<uint32_t>(s) < N;
            bad |= !ok;
            unsorted |= (e % kr) > 0 && __ldg(a.idx_r + tok0 * kr + e - 1) >= s;
            s_ir[e] = s;
            s_wr[e] = ok ? __ldg(a.w_r + tok0 * kr + e) : 0.f;
        }
        for (int t = tid; t < n; t += CK_THREADS) {
            const float al = load_elem<D>(a.alpha, tok0 + t);
            s_al[t] = al;
            // log(alpha) floored at -80 (e^-80 < 2^-115): a gate of exactly 0, which the fp32
            // gate formula reaches for large A softplus(.), then decays to below fp32 precision
            // of any stored value instead of making lam = -inf and exp(-inf - -inf) = NaN
            s_la[t] = al > 0.f ? fmaxf(logf(al), -80.f) : -80.f;
            s_be[t] = load_elem<D>(a.beta, tok0 + t);
        }
        for (int e = tid; e < n * dv; e += CK_THREADS) s_dV[e] = load_elem<D>(a.v, tok0 * dv + e);
        __syncthreads();
        // ---- S1: segmented cumulative log-decays
        for (int e = tid; e < n * (kw + kr); e += CK_THREADS) {
            const bool w_side = e < n * kw;
            const int q = w_side ? e : e - n * kw;
            const int k = w_side ? kw : kr;
            const int t = q / k;
            const int s = w_side ? s_iw[q] : s_ir[q];
            float lam = 0.f;
            for (int u = 0; u <= t; ++u)
                if (find_slot(s_iw + u * kw, kw, s) >= 0) lam += s_la[u];
            (w_side ? s_lw : s_lr)[q] = lam;
        }
        __syncthreads();
        // ---- S2: interaction matrices
        for (int p = tid; p < n * n; p += CK_THREADS) {
            const int t = p / n, s = p - t * n;
            s_A[t * C + s] = s < t ? gated_ip(s_iw + t * kw, s_ww + t * kw, s_lw + t * kw, kw, s_iw + s * kw,
                                              s_ww + s * kw, s_lw + s * kw, kw)
                                   : 0.f;
            s_QK[t * C + s] = s <= t ? gated_ip(s_ir + t * kr, s_wr + t * kr, s_lr + t * kr, kr, s_iw + s * kw,
                                                s_ww + s * kw, s_lw + s * kw, kw)
                                     : 0.f;
        }
        __syncthreads();
        // ---- S3: forward substitution, row by row: dV[t] = beta_t (v_t - sum_{s<t} A[t][s] dV[s]),
        //      B[t][j] = -beta_t (delta_tj + sum_{s<t} A[t][s] B[s][j])
        for (int t = 0; t < n; ++t) {
            const float bt = s_be[t];
            for (int col = tid; col < dv + n; col += CK_THREADS) {
                if (col < dv) {
                    float acc = s_dV[t * dv + col];
                    for (int s = 0; s < t; ++s) acc = fmaf(-s_A[t * C + s], s_dV[s * dv + col], acc);
                    s_dV[t * dv + col] = bt * acc;
                } else {
                    const int j = col - dv;
                    float acc = j == t ? 1.f : 0.f;
                    for (int s = 0; s < t; ++s) acc = fmaf(s_A[t * C + s], s_B[s * C + j], acc);
                    s_B[t * C + j] = -bt * acc;
                }
            }
            __syncthreads();
        }
        // ---- S4: gathers from the chunk-initial memory: one thread per (token, 16-byte piece of
        //      the row), 16-byte loads, four rows in flight
        {
            constexpr int E = D::E;
            const int npc = dv / E;                                   // 16-byte pieces per row
            const char* mrows = static_cast<const char*>(a.mem) + mrow0 * dv * D::BYTES;
            for (int e = tid; e < n * npc; e += CK_THREADS) {
                const int t = e / npc, c = e - t * npc;
                float rv[E], iv[E];
#pragma unroll
                for (int j = 0; j < E; ++j) { rv[j] = 0.f; iv[j] = 0.f; }
                auto acc_rows = [&](const int* sl, const float* sw, const float* slam, int k, float (&out)[E]) {
                    for (int m0 = 0; m0 < k; m0 += 4) {
                        uint4 raw[4];
                        float cf[4];
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int m = m0 + q;
                            const int s = m < k ? sl[t * k + m] : -1;
                            const bool ok = m < k && static_cast<uint32_t>(s) < N;
                            cf[q] = ok ? sw[t * k + m] * __expf(slam[t * k + m]) : 0.f;
                            raw[q] = ok ? __ldg(reinterpret_cast<const uint4*>(mrows + (static_cast<int64_t>(s) * dv) * D::BYTES) + c)
                                        : make_uint4(0u, 0u, 0u, 0u);
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            float f[E];
                            unpack16<D>(raw[q], f);
#pragma unroll
                            for (int j = 0; j < E; ++j) out[j] = fmaf(cf[q], f[j], out[j]);
                        }
                    }
                };
                acc_rows(s_iw, s_ww, s_lw, kw, rv);
                acc_rows(s_ir, s_wr, s_lr, kr, iv);
#pragma unroll
                for (int j = 0; j < E; ++j) {
                    s_R[t * dv + c * E + j] = rv[j];
                    s_I[t * dv + c * E + j] = iv[j];
                }
            }
        }
        __syncthreads();
        // ---- S5: u = dV + B retrieved (in place, rows descending), then y = inter + QK u
        for (int d = tid; d < dv; d += CK_THREADS) {
            for (int t = n - 1; t >= 0; --t) {
                float acc = s_dV[t * dv + d];
                for (int s = 0; s <= t; ++s) acc = fmaf(s_B[t * C + s], s_R[s * dv + d], acc);
                s_R[t * dv + d] = acc;
            }
            for (int t = 0; t < n; ++t) {
                float acc = s_I[t * dv + d];
                for (int s = 0; s <= t; ++s) acc = fmaf(s_QK[t * C + s], s_R[s * dv + d], acc);
                store_val<D>(a.y, (tok0 + t) * dv + d, acc);
            }
        }
        __syncthreads();
        // ---- S6: one warp per write entry that is its slot's last occurrence in the chunk
        for (int e = warp; e < n * kw; e += CK_THREADS / 32) {
            const int t = e / kw;
            const int s = s_iw[e];
            if (static_cast<uint32_t>(s) >= N) continue;               // warp-uniform
            // later writers of s in the chunk (lane u checks token t + 1 + u)
            const int u_late = t + 1 + lane;
            const bool later = u_late < n && find_slot(s_iw + u_late * kw, kw, s) >= 0;
            if (__any_sync(0xffffffffu, later)) continue;
            // occurrences of s among tokens 0..t (lane u checks token u; n <= 32)
            const int pos = lane <= t ? find_slot(s_iw + lane * kw, kw, s) : -1;
            const uint32_t occ = __ballot_sync(0xffffffffu, pos >= 0);
            const float lam = s_lw[e];                                  // the slot's decay over the chunk
            const float dec = __expf(lam);
            float acc[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int d = lane + 32 * j;
                acc[j] = d < dv ? dec * load_elem<D>(a.mem, (mrow0 + s) * dv + d) : 0.f;
            }
            uint32_t mask = occ;
            while (mask) {                                              // warp-uniform
                const int u = __ffs(mask) - 1;
                mask &= mask - 1;
                const int pu = __shfl_sync(0xffffffffu, pos, u);
                const float cf = __expf(lam - s_lw[u * kw + pu]) * s_ww[u * kw + pu];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int d = lane + 32 * j;
                    if (d < dv) acc[j] = fmaf(cf, s_R[u * dv + d], acc[j]);
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int d = lane + 32 * j;
                if (d < dv) store_val<D>(a.mem, (mrow0 + s) * dv + d, acc[j]);
            }
        }
        __syncthreads();
    }
    if (bad && (threadIdx.x & 31) == 0) flag_error(a.err, ERR_BAD_INDEX);
    if (unsorted) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_recur_chunkwise(int dtype, const RecArgs& a, int C, cudaStream_t stream) {
    const size_t smem = chunk_smem_bytes(C, a.kw, a.kr, a.dv);
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    if (dtype == 0) {
        cudaError_t e = cudaFuncSetAttribute(k_recur_chunk<F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_recur_chunk<F32><<<static_cast<unsigned>(chains), CK_THREADS, smem, stream>>>(a, C);
    } else {
        cudaError_t e = cudaFuncSetAttribute(k_recur_chunk<BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_recur_chunk<BF16><<<static_cast<unsigned>(chains), CK_THREADS, smem, stream>>>(a, C);
    }
    return cudaGetLastError();
}

}  // namespace sdm
