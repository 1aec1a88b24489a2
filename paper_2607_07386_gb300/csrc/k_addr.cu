// K-ADDR: sparse key selection (Sec. 3.1 item 1; Sec. 2 "Product Key Memory"; Sec. 4 softmax).
//
// For every token x (k for the write side, q for the read side) of head h:
//   s = P_h x in R^{2S} (PROJECTED) or s = x (DIRECT, d_k = 2S); s1 = s[0:S], s2 = s[S:2S];
//   T1 = top_k(s1), T2 = top_k(s2) under (score desc, index asc);
//   slots = top_k over (i, j) in T1 x T2 of s1[i] + s2[j] under (score desc, slot asc),
//           slot = i*S + j  (the PKM identity of Sec. 2 makes this the top-k of all N);
//   w = softmax of the selected scores; output sorted ascending by slot (App. A.2).
//
// Exactness.  The selected SETS must equal those of the float64 definition.  Scores are
// computed in fp32 with a rigorous error bound eps = cbound * max_j ||P_j|| * ||x||
// (Cauchy-Schwarz on the accumulation error bound gamma_dk * sum |P_jd x_d|).  A top-k
// boundary is certified when the gap between the k-th and (k+1)-th fp32 values exceeds
// 2 eps; otherwise the entries inside the uncertainty band are re-scored in float64 with
// the sequential ascending-d order (bit-identical to the float64 definition: products of
// two storage numbers are exact in float64) and re-decided.  Each chunk keeps the top
// L = k + margin entries so the band is normally inside the list; if it is not, the
// whole half (or all k^2 candidates) is recomputed in float64.
//
// Kernel A (k_addr_scores): one CTA = 128 tokens of one head x one column chunk; one
//   thread per token accumulates 32 columns at a time in fp32 FFMA (fixed d order) and
//   keeps a sorted top-L list; lists go to the workspace.
// Kernel B (k_addr_finalize): one thread per token merges the chunk lists of each half,
//   certifies both halves, enumerates the outer-sum candidates above a provable
//   threshold, certifies the combined boundary, applies softmax and sorts by slot.
#include "sdm_internal.h"

#include <float.h>

namespace sdm {

constexpr int A_TOK = 128;     // tokens per score CTA (one per thread)
constexpr int A_SUB = 32;      // columns accumulated per pass
constexpr int A_PPITCH = 36;   // fp32 pitch of the staged P sub-chunk (16-byte aligned, fewer bank conflicts)
constexpr int F_THREADS = 64;  // tokens per finalize CTA (wide lists)
constexpr int FW_WARPS = 8;    // warps (= token-sides) per finalize CTA (k <= 32)

// Per-chunk top-L lists: entry p of token u, chunk `chunk` of (side, head) z is at
// ((z * 2 ncc + chunk) * BT + u) * L + p  (a token's L entries are contiguous).
__host__ __device__ __forceinline__ int64_t part_at(int z, int ncc, int chunk, int64_t BT, int64_t u, int L, int p) {
    return ((static_cast<int64_t>(z) * (2 * ncc) + chunk) * BT + u) * L + p;
}

// Sorted (value desc, index asc) list of the L best entries seen so far; empty = -inf.
template <int L>
struct TopList {
    float v[L];
    int i[L];
    __device__ __forceinline__ void clear() {
#pragma unroll
        for (int p = 0; p < L; ++p) { v[p] = -INFINITY; i[p] = INT_MAX; }
    }
    __device__ __forceinline__ static bool beats(float a, int ia, float b, int ib) {
        return (a > b) || (a == b && ia < ib);
    }
    __device__ __forceinline__ bool admits(float x, int ix) const { return beats(x, ix, v[L - 1], i[L - 1]); }
    // General insertion (caller checked admits()).
    __device__ __forceinline__ void push(float x, int ix) {
#pragma unroll
        for (int p = 0; p < L; ++p) {
            const bool b = beats(x, ix, v[p], i[p]);
            const float tv = v[p];
            const int ti = i[p];
            v[p] = b ? x : tv; i[p] = b ? ix : ti;
            x = b ? tv : x;   ix = b ? ti : ix;
        }
    }
    // Insertion when every present entry has a smaller index than ix (scan order):
    // equal values never move, so a strict compare suffices.
    __device__ __forceinline__ void push_scan(float x, int ix) {
#pragma unroll
        for (int p = 0; p < L; ++p) {
            const bool b = x > v[p];
            const float tv = v[p];
            const int ti = i[p];
            v[p] = b ? x : tv; i[p] = b ? ix : ti;
            x = b ? tv : x;   ix = b ? ti : ix;
        }
    }
};

template <int L>
__device__ __forceinline__ float pick(const float (&a)[L], int p) {
    float r = a[0];
#pragma unroll
    for (int q = 1; q < L; ++q) r = (q == p) ? a[q] : r;
    return r;
}

// ------------------------------------------------------------------------------------------
// Kernel A: fp32 half-scores + per-chunk top-L
// ------------------------------------------------------------------------------------------
template <class D, int L>
__global__ void __launch_bounds__(A_TOK) k_addr_scores(const AddrArgs a) {
    extern __shared__ __align__(16) float smA[];
    float* xs = smA;                               // [dk][A_TOK]  x of the CTA's tokens, transposed
    float* ps = smA + a.dk * A_TOK;                // [dk][A_PPITCH] staged P rows of one sub-chunk
    const int tid = threadIdx.x;
    const int which = blockIdx.z / a.H, h = blockIdx.z % a.H;
    const int chunk = blockIdx.y;
    const int hf = chunk / a.ncc, cc = chunk % a.ncc;
    const int c0 = cc * a.cw, c1 = min(a.S, c0 + a.cw);
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    const int64_t u0 = static_cast<int64_t>(blockIdx.x) * A_TOK;
    const void* X = a.X[which];
    const void* P = a.P[which];

    for (int e = tid; e < A_TOK * a.dk; e += A_TOK) {
        const int ul = e / a.dk, d = e - ul * a.dk;
        const int64_t u = u0 + ul;
        float val = 0.f;
        if (u < BT) {
            const int64_t b = u / a.T, t = u - b * a.T;
            val = load_elem<D>(X, ((b * a.H + h) * a.T + t) * a.dk + d);
        }
        xs[d * A_TOK + ul] = val;
    }

    TopList<L> top;
    top.clear();
    const int64_t prow0 = static_cast<int64_t>(h) * 2 * a.S + static_cast<int64_t>(hf) * a.S;
    for (int s0 = c0; s0 < c1; s0 += A_SUB) {
        __syncthreads();   // xs staged / previous sub-chunk consumed
        float acc[A_SUB];
        if (P == nullptr) {
#pragma unroll
            for (int jj = 0; jj < A_SUB; ++jj) {
                const int col = s0 + jj;
                acc[jj] = (col < c1) ? xs[(hf * a.S + col) * A_TOK + tid] : -INFINITY;
            }
        } else {
            for (int e = tid; e < A_SUB * a.dk; e += A_TOK) {
                const int jj = e / a.dk, d = e - jj * a.dk;
                const int col = s0 + jj;
                ps[d * A_PPITCH + jj] = (col < c1) ? load_elem<D>(P, (prow0 + col) * a.dk + d) : 0.f;
            }
            __syncthreads();
#pragma unroll
            for (int jj = 0; jj < A_SUB; ++jj) acc[jj] = 0.f;
            for (int d = 0; d < a.dk; ++d) {            // ascending d, one rounding per step
                const float xv = xs[d * A_TOK + tid];
                const float4* pr = reinterpret_cast<const float4*>(ps + d * A_PPITCH);
#pragma unroll
                for (int q = 0; q < A_SUB / 4; ++q) {
                    const float4 p4 = pr[q];
                    acc[4 * q + 0] = fmaf(xv, p4.x, acc[4 * q + 0]);
                    acc[4 * q + 1] = fmaf(xv, p4.y, acc[4 * q + 1]);
                    acc[4 * q + 2] = fmaf(xv, p4.z, acc[4 * q + 2]);
                    acc[4 * q + 3] = fmaf(xv, p4.w, acc[4 * q + 3]);
                }
            }
        }
#pragma unroll
        for (int jj = 0; jj < A_SUB; ++jj) {
            const int col = s0 + jj;
            if (col < c1 && acc[jj] > top.v[L - 1]) top.push_scan(acc[jj], col);
        }
    }

    const int64_t u = u0 + tid;
    if (u < BT) {
        const int64_t base = part_at(blockIdx.z, a.ncc, chunk, BT, u, L, 0);
#pragma unroll
        for (int p = 0; p < L; ++p) {
            a.part_v[base + p] = top.v[p];
            a.part_i[base + p] = top.i[p];
        }
    }
}

// ------------------------------------------------------------------------------------------
// Kernel B helpers
// ------------------------------------------------------------------------------------------
struct TokenCtx {
    int* err;           // device status word / counters
    const void* P;      // P of this side (nullptr = DIRECT)
    const void* X;
    int64_t xoff;       // element offset of the token's x row
    int64_t prow0;      // row of P for column 0 of half 0 (= h * 2S)
    int dk, S;
};

// Float64 score of column j of half hf, summed over d in ascending order.
template <class D>
__device__ double score64(const TokenCtx& c, int hf, int j) {
    if (c.P == nullptr) return static_cast<double>(load_elem<D>(c.X, c.xoff + static_cast<int64_t>(hf) * c.S + j));
    const int64_t prow = (c.prow0 + static_cast<int64_t>(hf) * c.S + j) * c.dk;
    double acc = 0.0;
    for (int d = 0; d < c.dk; ++d)
        acc = fma(static_cast<double>(load_elem<D>(c.P, prow + d)), static_cast<double>(load_elem<D>(c.X, c.xoff + d)), acc);
    return acc;
}

__device__ __forceinline__ bool beats64(double a, int ia, double b, int ib) { return (a > b) || (a == b && ia < ib); }

// Uncertified half boundary: decide the band in float64.  lv/li: top-L by fp32 (sorted).
// Writes the exact top-k (ordered by fp32 value, desc) to Av/Ai with pitch F_THREADS.
template <class D, int L>
__device__ __noinline__ void resolve_half(const float* lv, const int* li, int k, double eps, const TokenCtx& c, int hf,
                                          float* Av, int* Ai, int pitch) {
    const double lo = static_cast<double>(lv[k - 1]) - 2.0 * eps;
    const double hi = static_cast<double>(lv[k]) + 2.0 * eps;
    if (c.S > L && static_cast<double>(lv[L - 1]) >= lo) {
        // Band may extend past the list: exact top-k of the whole half in float64.
        stat_add(c.err, STAT_HALF_FULL);
        double bv[64 + 4];
        int bi[64 + 4];
        int n = 0;
        for (int j = 0; j < c.S; ++j) {
            const double s = score64<D>(c, hf, j);
            if (n == k && !beats64(s, j, bv[k - 1], bi[k - 1])) continue;
            int p = (n < k) ? n++ : k - 1;
            while (p > 0 && beats64(s, j, bv[p - 1], bi[p - 1])) { bv[p] = bv[p - 1]; bi[p] = bi[p - 1]; --p; }
            bv[p] = s; bi[p] = j;
        }
        for (int p = 0; p < k; ++p) { Av[p * pitch] = static_cast<float>(bv[p]); Ai[p * pitch] = bi[p]; }
        return;
    }
    stat_add(c.err, STAT_BAND_F64);
    int cin = 0;
    while (cin < L && static_cast<double>(lv[cin]) > hi) ++cin;
    int pend = cin;
    while (pend < L && static_cast<double>(lv[pend]) >= lo) ++pend;
    double s64[L];
    bool used[L];
    for (int p = cin; p < pend; ++p) { s64[p] = score64<D>(c, hf, li[p]); used[p] = false; }
    for (int p = 0; p < cin; ++p) { Av[p * pitch] = lv[p]; Ai[p * pitch] = li[p]; }
    // choose k - cin entries of the band by (float64 desc, index asc) ...
    int chosen[L];
    const int need = k - cin;
    for (int r = 0; r < need; ++r) {
        int best = -1;
        for (int p = cin; p < pend; ++p)
            if (!used[p] && (best < 0 || beats64(s64[p], li[p], s64[best], li[best]))) best = p;
        used[best] = true;
        chosen[r] = best;
    }
    // ... and keep them in fp32-value order (they all lie below the certain entries)
    for (int r = 0; r < need; ++r) {
        int best = -1;
        for (int q = 0; q < need; ++q) {
            const int p = chosen[q];
            if (p >= 0 && (best < 0 || TopList<L>::beats(lv[p], li[p], lv[chosen[best]], li[chosen[best]]))) best = q;
        }
        Av[(cin + r) * pitch] = lv[chosen[best]];
        Ai[(cin + r) * pitch] = li[chosen[best]];
        chosen[best] = -1;
    }
}

// Uncertified combined boundary.  cv/cf: top-L candidates by fp32 (sorted).  A1/A2: the two
// exact half lists.  Writes the exact top-k (fp32 score, slot) to Fv/Fi.
template <class D, int L>
__device__ __noinline__ void resolve_combined(const float* cv, const int* cf, int k, double epsc, const TokenCtx& c,
                                              const float* A1v, const int* A1i, const float* A2v, const int* A2i,
                                              float* Fv, int* Fi, int pitch) {
    const int S = c.S;
    const double lo = static_cast<double>(cv[k - 1]) - 2.0 * epsc;
    const double hi = static_cast<double>(cv[k]) + 2.0 * epsc;
    if (cv[L - 1] != -INFINITY && static_cast<double>(cv[L - 1]) >= lo) {
        // All k^2 candidates in float64.
        stat_add(c.err, STAT_COMB_FULL);
        double s1[64], s2[64];
        for (int p = 0; p < k; ++p) { s1[p] = score64<D>(c, 0, A1i[p * pitch]); s2[p] = score64<D>(c, 1, A2i[p * pitch]); }
        double bv[64];
        int bf[64], bp1[64], bp2[64];
        int n = 0;
        for (int p1 = 0; p1 < k; ++p1)
            for (int p2 = 0; p2 < k; ++p2) {
                const double s = s1[p1] + s2[p2];
                const int f = A1i[p1 * pitch] * S + A2i[p2 * pitch];
                if (n == k && !beats64(s, f, bv[k - 1], bf[k - 1])) continue;
                int p = (n < k) ? n++ : k - 1;
                while (p > 0 && beats64(s, f, bv[p - 1], bf[p - 1])) {
                    bv[p] = bv[p - 1]; bf[p] = bf[p - 1]; bp1[p] = bp1[p - 1]; bp2[p] = bp2[p - 1]; --p;
                }
                bv[p] = s; bf[p] = f; bp1[p] = p1; bp2[p] = p2;
            }
        for (int p = 0; p < k; ++p) {
            Fv[p * pitch] = A1v[bp1[p] * pitch] + A2v[bp2[p] * pitch];
            Fi[p * pitch] = bf[p];
        }
        return;
    }
    stat_add(c.err, STAT_BAND_F64);
    int cin = 0;
    while (cin < L && static_cast<double>(cv[cin]) > hi) ++cin;
    int pend = cin;
    while (pend < L && static_cast<double>(cv[pend]) >= lo) ++pend;
    double s64[L];
    bool used[L];
    for (int p = cin; p < pend; ++p) {
        s64[p] = score64<D>(c, 0, cf[p] / S) + score64<D>(c, 1, cf[p] % S);
        used[p] = false;
    }
    for (int p = 0; p < cin; ++p) { Fv[p * pitch] = cv[p]; Fi[p * pitch] = cf[p]; }
    for (int r = cin; r < k; ++r) {
        int best = -1;
        for (int p = cin; p < pend; ++p)
            if (!used[p] && (best < 0 || beats64(s64[p], cf[p], s64[best], cf[best]))) best = p;
        used[best] = true;
        Fv[r * pitch] = cv[best];
        Fi[r * pitch] = cf[best];
    }
}

// ------------------------------------------------------------------------------------------
// Kernel B (k <= 32): one warp per token-side.  Lane p holds entry p (and p + 32) of a list.
//   merge of chunk lists: output rank = own position + number of entries of the other list
//     that come first (binary search across lanes), scattered through shared memory;
//   combined top-(k+4): exact k-way merge of the k rows i of the outer sum (lane i owns row
//     i, its head s1[i] + s2[j_i]); each step takes the largest head by a warp max-reduce of
//     order-preserving integer keys, ties to the smallest slot by a min-reduce;
//   softmax by warp reductions; ascending slot order by a 32-lane bitonic shuffle network.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t f2key(float f) {
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key2f(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// entry idx (< 64) of a list held two entries per lane (v0: idx < 32, v1: idx >= 32)
__device__ __forceinline__ float lane_get(float v0, float v1, int idx) {
    const float a = __shfl_sync(0xffffffffu, v0, idx & 31);
    const float b = __shfl_sync(0xffffffffu, v1, idx & 31);
    return idx < 32 ? a : b;
}
// number of the first L entries of a descending list that are > x (strict) or >= x
__device__ __forceinline__ int lane_count_before(float v0, float v1, int L, float x, bool strict) {
    int pos = 0;
#pragma unroll
    for (int step = 32; step >= 1; step >>= 1) {
        const int idx = pos + step - 1;
        const float v = lane_get(v0, v1, idx);
        const bool before = strict ? (v > x) : (v >= x);
        if (idx < L && before) pos += step;
    }
    return pos;
}

__device__ __forceinline__ int lane_geti(int i0, int i1, int idx) {
    const int a = __shfl_sync(0xffffffffu, i0, idx & 31);
    const int b = __shfl_sync(0xffffffffu, i1, idx & 31);
    return idx < 32 ? a : b;
}

// Compensated fp32 score of column j of half hf (one lane, one column).  Every product is
// split exactly (p + pe = P x, pe = 0 for bf16 operands) and every addition exactly by
// TwoSum (s + err = s_old + p); the error terms are summed in plain fp32.  With n = d_k
// terms and u = 2^-24 the result val = s + e differs from the exact dot product by at
// most 2 n (n + 1) u^2 (1.03) sum|P x| <= 2^-31 sum|P x| for n <= 256.  The float64
// sequential sum of the definition lies within (n - 1) 2^-53 sum|P x| of the exact value,
// so `bound` = 2^-28 sum|P x| (+ 2^-50 |val| for the conversion to double) covers the
// distance to it with margin.  DIRECT addressing: the score is x itself, exact (bound 0).
template <class D>
__device__ void ff_score(const TokenCtx& c, int hf, int j, double& val, double& bound) {
    if (c.P == nullptr) {
        val = static_cast<double>(load_elem<D>(c.X, c.xoff + static_cast<int64_t>(hf) * c.S + j));
        bound = 0.0;
        return;
    }
    const int64_t prow = (c.prow0 + static_cast<int64_t>(hf) * c.S + j) * c.dk;
    float sum = 0.f, err = 0.f, mag = 0.f;
#pragma unroll 8
    for (int d = 0; d < c.dk; ++d) {
        const float pv = load_elem<D>(c.P, prow + d);
        const float xv = load_elem<D>(c.X, c.xoff + d);
        const float p = __fmul_rn(pv, xv);
        const float pe = __fmaf_rn(pv, xv, -p);
        const float t = __fadd_rn(sum, p);
        const float bp = __fsub_rn(t, sum);
        const float e2 = __fadd_rn(__fsub_rn(sum, __fsub_rn(t, bp)), __fsub_rn(p, bp));
        sum = t;
        err = __fadd_rn(err, __fadd_rn(e2, pe));
        mag = __fadd_rn(mag, fabsf(p));
    }
    val = static_cast<double>(sum) + static_cast<double>(err);
    bound = 0x1p-28 * static_cast<double>(mag) + 0x1p-50 * fabs(val);
}

// Band entries [cin, cin + m) of a list sorted by fp32 score are re-ranked by their
// compensated scores (one lane per entry).  Returns false when two entries are closer
// than their bounds (the float64 definition must decide) -- otherwise the ranks are
// those of the float64 definition under (score desc, index asc).
__device__ __forceinline__ bool rank_band(double cd, double eb, int id, int m, int lane, int& rank) {
    rank = 0;
    bool unsure = false;
    for (int f = 0; f < m; ++f) {
        const double cf = __shfl_sync(0xffffffffu, cd, f);
        const double ef = __shfl_sync(0xffffffffu, eb, f);
        const int jf = __shfl_sync(0xffffffffu, id, f);
        if (lane < m && f != lane) {
            const double tol = ef + eb;
            const double diff = cf - cd;
            if (tol > 0.0 && fabs(diff) <= tol) unsure = true;
            else rank += (diff > 0.0 || (diff == 0.0 && jf < id)) ? 1 : 0;
        }
    }
    return !__any_sync(0xffffffffu, unsure);
}

// Warp-cooperative resolution of an uncertified half boundary (list: lane p holds entry p
// in v0/i0 and entry p + 32 in v1/i1).  On success writes the exact top-k, in fp32-list
// order, to ov/oi[0, k) and returns true; returns false when the serial float64 path must
// decide (band past the list, more than 32 band entries, or an unresolved near-tie).
template <class D, int L>
__device__ bool warp_band_half(float v0, int i0, float v1, int i1, int k, double eps, const TokenCtx& c, int hf,
                               float* ov, int* oi, int lane) {
    const double lo = static_cast<double>(lane_get(v0, v1, k - 1)) - 2.0 * eps;
    const double hi = static_cast<double>(lane_get(v0, v1, k)) + 2.0 * eps;
    if (c.S > L && static_cast<double>(lane_get(v0, v1, L - 1)) >= lo) return false;
    const double d0 = static_cast<double>(v0), d1 = static_cast<double>(v1);
    const int cin = __popc(__ballot_sync(0xffffffffu, lane < L && d0 > hi)) +
                    __popc(__ballot_sync(0xffffffffu, lane + 32 < L && d1 > hi));
    const int m = __popc(__ballot_sync(0xffffffffu, lane < L && d0 >= lo && d0 <= hi)) +
                  __popc(__ballot_sync(0xffffffffu, lane + 32 < L && d1 >= lo && d1 <= hi));
    if (m > 32) return false;
    const int p = min(cin + lane, L - 1);
    const float bv = lane_get(v0, v1, p);
    const int bi = lane_geti(i0, i1, p);
    double cd = 0.0, eb = 0.0;
    if (lane < m) ff_score<D>(c, hf, bi, cd, eb);
    int rank;
    if (!rank_band(cd, eb, bi, m, lane, rank)) return false;
    const bool chosen = lane < m && rank < k - cin;
    const unsigned ch = __ballot_sync(0xffffffffu, chosen);
    __syncwarp();
    if (lane < cin) { ov[lane] = v0; oi[lane] = i0; }
    if (chosen) {
        const int q = cin + __popc(ch & ((1u << lane) - 1u));
        ov[q] = bv;
        oi[q] = bi;
    }
    __syncwarp();
    return true;
}

// Same for the outer-sum boundary: candidate slot f = i S + j is rescored as the sum of
// the compensated half scores of column i (half 0) and column j (half 1).  The float64
// definition adds its two half scores with one more rounding (<= 2^-53 of the sum).
template <class D, int L>
__device__ bool warp_band_comb(float v0, int f0, float v1, int f1, int k, double epsc, const TokenCtx& c,
                               float* ov, int* oi, int lane) {
    const double lo = static_cast<double>(lane_get(v0, v1, k - 1)) - 2.0 * epsc;
    const double hi = static_cast<double>(lane_get(v0, v1, k)) + 2.0 * epsc;
    const float vl = lane_get(v0, v1, L - 1);
    if (vl != -INFINITY && static_cast<double>(vl) >= lo) return false;
    const double d0 = static_cast<double>(v0), d1 = static_cast<double>(v1);
    const int cin = __popc(__ballot_sync(0xffffffffu, lane < L && d0 > hi)) +
                    __popc(__ballot_sync(0xffffffffu, lane + 32 < L && d1 > hi));
    const int m = __popc(__ballot_sync(0xffffffffu, lane < L && d0 >= lo && d0 <= hi)) +
                  __popc(__ballot_sync(0xffffffffu, lane + 32 < L && d1 >= lo && d1 <= hi));
    if (m > 32) return false;
    const int p = min(cin + lane, L - 1);
    const float bv = lane_get(v0, v1, p);
    const int bf = lane_geti(f0, f1, p);
    double cd = 0.0, eb = 0.0;
    if (lane < m) {
        double c1, e1, c2, e2;
        ff_score<D>(c, 0, bf / c.S, c1, e1);
        ff_score<D>(c, 1, bf % c.S, c2, e2);
        cd = c1 + c2;
        eb = (c.P == nullptr) ? 0.0 : e1 + e2 + 0x1p-50 * fabs(cd);
    }
    int rank;
    if (!rank_band(cd, eb, bf, m, lane, rank)) return false;
    const bool chosen = lane < m && rank < k - cin;
    const unsigned ch = __ballot_sync(0xffffffffu, chosen);
    __syncwarp();
    if (lane < cin) { ov[lane] = v0; oi[lane] = f0; }
    if (chosen) {
        const int q = cin + __popc(ch & ((1u << lane) - 1u));
        ov[q] = bv;
        oi[q] = bf;
    }
    __syncwarp();
    return true;
}

template <class D, int L>
__global__ void __launch_bounds__(FW_WARPS * 32) k_addr_finalize(const AddrArgs a) {
    static_assert(L <= 36, "warp finalize handles k <= 32");
    __shared__ float wv[FW_WARPS][3][64];
    __shared__ int wi[FW_WARPS][3][64];
    const int lane = threadIdx.x & 31, wq = threadIdx.x >> 5;
    const int z = blockIdx.y;
    const int side = z / a.H, h = z % a.H;
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    const int64_t u = static_cast<int64_t>(blockIdx.x) * FW_WARPS + wq;
    if (u >= BT) return;                                   // whole warp
    const int k = a.kk[side];
    const int S = a.S;
    const int64_t b = u / a.T, t = u - b * a.T;
    TokenCtx c;
    c.err = a.err;
    c.P = a.P[side];
    c.X = a.X[side];
    c.xoff = ((b * a.H + h) * a.T + t) * a.dk;
    c.prow0 = static_cast<int64_t>(h) * 2 * S;
    c.dk = a.dk;
    c.S = S;
    float* sv0 = wv[wq][0]; int* si0 = wi[wq][0];          // staging / merge output / A1
    float* sv1 = wv[wq][1]; int* si1 = wi[wq][1];          // A2
    float* sv2 = wv[wq][2]; int* si2 = wi[wq][2];          // candidates / final

    double eps = 0.0;
    if (c.P != nullptr) {
        float ss = 0.f;
        for (int d = lane; d < a.dk; d += 32) {
            const float xv = load_elem<D>(c.X, c.xoff + d);
            ss = fmaf(xv, xv, ss);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        eps = static_cast<double>(a.cbound) * static_cast<double>(a.pnorm[side * a.H + h]) *
              static_cast<double>(sqrtf(ss)) * (1.0 + 0x1p-12);
    }

    float av[2], bv[2];      // A1 and A2 after certification: lane p holds entry p (p < k)
    int ai[2], bi[2];
    float amax[2];
#pragma unroll 1
    for (int hf = 0; hf < 2; ++hf) {
        // chunk 0 of this half
        int64_t base = part_at(z, a.ncc, hf * a.ncc, BT, u, L, 0);
        float v0 = lane < L ? a.part_v[base + lane] : -INFINITY;
        float v1 = lane + 32 < L ? a.part_v[base + lane + 32] : -INFINITY;
        int i0 = lane < L ? a.part_i[base + lane] : INT_MAX;
        int i1 = lane + 32 < L ? a.part_i[base + lane + 32] : INT_MAX;
        for (int cc = 1; cc < a.ncc; ++cc) {                  // merge later chunks (larger columns)
            base = part_at(z, a.ncc, hf * a.ncc + cc, BT, u, L, 0);
            const float w0 = lane < L ? a.part_v[base + lane] : -INFINITY;
            const float w1 = lane + 32 < L ? a.part_v[base + lane + 32] : -INFINITY;
            const int j0 = lane < L ? a.part_i[base + lane] : INT_MAX;
            const int j1 = lane + 32 < L ? a.part_i[base + lane + 32] : INT_MAX;
            // ties: the earlier chunk first
            const int ra0 = lane + lane_count_before(w0, w1, L, v0, true);
            const int ra1 = lane + 32 + lane_count_before(w0, w1, L, v1, true);
            const int rb0 = lane + lane_count_before(v0, v1, L, w0, false);
            const int rb1 = lane + 32 + lane_count_before(v0, v1, L, w1, false);
            __syncwarp();
            if (lane < L && ra0 < L) { sv0[ra0] = v0; si0[ra0] = i0; }
            if (lane + 32 < L && ra1 < L) { sv0[ra1] = v1; si0[ra1] = i1; }
            if (lane < L && rb0 < L) { sv0[rb0] = w0; si0[rb0] = j0; }
            if (lane + 32 < L && rb1 < L) { sv0[rb1] = w1; si0[rb1] = j1; }
            __syncwarp();
            v0 = lane < L ? sv0[lane] : -INFINITY;       i0 = lane < L ? si0[lane] : INT_MAX;
            v1 = lane + 32 < L ? sv0[lane + 32] : -INFINITY; i1 = lane + 32 < L ? si0[lane + 32] : INT_MAX;
        }
        // certify the boundary between entries k-1 and k (warp-uniform decision)
        bool certified = S <= k;
        if (!certified) {
            const float vk = lane_get(v0, v1, k - 1), vk1 = lane_get(v0, v1, k);
            certified = static_cast<double>(vk) - static_cast<double>(vk1) > 2.0 * eps;
        }
        if (!certified) {
            if (lane == 0) stat_add(c.err, STAT_HALF_BAND);
            if (!warp_band_half<D, L>(v0, i0, v1, i1, k, eps, c, hf, sv0, si0, lane)) {
                __syncwarp();
                if (lane < L) { sv0[lane] = v0; si0[lane] = i0; }
                if (lane + 32 < L) { sv0[lane + 32] = v1; si0[lane + 32] = i1; }
                __syncwarp();
                if (lane == 0) {
                    float lv[L];
                    int li[L];
                    for (int p = 0; p < L; ++p) { lv[p] = sv0[p]; li[p] = si0[p]; }
                    resolve_half<D, L>(lv, li, k, eps, c, hf, sv0, si0, 1);
                }
            }
            __syncwarp();
            v0 = lane < k ? sv0[lane] : -INFINITY;
            i0 = lane < k ? si0[lane] : INT_MAX;
        }
        if (hf == 0) { av[0] = lane < k ? v0 : -INFINITY; ai[0] = i0; }
        else { bv[0] = lane < k ? v0 : -INFINITY; bi[0] = i0; }
        amax[hf] = fmaxf(fabsf(lane_get(v0, v1, 0)), fabsf(lane_get(v0, v1, k - 1)));
    }

    // combined: k-way merge of the rows (lane i: row i; head = A1[i] + A2[j])
    const double epsc = 2.0 * eps + 0x1p-22 * (static_cast<double>(amax[0]) + static_cast<double>(amax[1]));
    int j = 0;
    const float b0v = __shfl_sync(0xffffffffu, bv[0], 0);
    const int b0i = __shfl_sync(0xffffffffu, bi[0], 0);
    float head = lane < k ? av[0] + b0v : -INFINITY;
    int flat = ai[0] * S + b0i;
    float cv0 = -INFINITY, cv1 = -INFINITY;    // candidate r in lane r (r < 32) / lane r-32
    int cf0 = INT_MAX, cf1 = INT_MAX;
    for (int r = 0; r < L; ++r) {
        const uint32_t key = f2key(head);
        const uint32_t kmax = __reduce_max_sync(0xffffffffu, key);
        const bool tie = key == kmax;
        const uint32_t fmin = __reduce_min_sync(0xffffffffu, tie ? static_cast<uint32_t>(flat) : 0xffffffffu);
        const bool win = tie && static_cast<uint32_t>(flat) == fmin;
        const float val = key2f(kmax);
        if (lane == (r & 31)) {
            if (r < 32) { cv0 = val; cf0 = static_cast<int>(fmin); }
            else { cv1 = val; cf1 = static_cast<int>(fmin); }
        }
        if (win) ++j;
        const float nv = __shfl_sync(0xffffffffu, bv[0], j & 31);
        const int ni = __shfl_sync(0xffffffffu, bi[0], j & 31);
        if (win) {
            head = (j < k && lane < k) ? av[0] + nv : -INFINITY;
            flat = ai[0] * S + ni;
        }
    }
    bool certified = (k == 1);
    if (!certified) {
        const float ck = lane_get(cv0, cv1, k - 1), ck1 = lane_get(cv0, cv1, k);
        certified = (ck1 == -INFINITY) || (static_cast<double>(ck) - static_cast<double>(ck1) > 2.0 * epsc);
    }
    float fv = cv0;
    int fi = cf0;
    if (!certified) {
        if (lane == 0) stat_add(c.err, STAT_COMB_BAND);
        if (!warp_band_comb<D, L>(cv0, cf0, cv1, cf1, k, epsc, c, sv2, si2, lane)) {
            __syncwarp();
            sv0[lane] = av[0]; si0[lane] = ai[0];            // A1
            sv1[lane] = bv[0]; si1[lane] = bi[0];            // A2
            sv2[lane] = cv0; si2[lane] = cf0;                // candidates 0..31
            if (lane + 32 < L) { sv2[lane + 32] = cv1; si2[lane + 32] = cf1; }
            __syncwarp();
            if (lane == 0) {
                float cvl[L];
                int cfl[L];
                for (int p = 0; p < L; ++p) { cvl[p] = sv2[p]; cfl[p] = si2[p]; }
                resolve_combined<D, L>(cvl, cfl, k, epsc, c, sv0, si0, sv1, si1, sv2, si2, 1);
            }
        }
        __syncwarp();
        fv = lane < k ? sv2[lane] : -INFINITY;
        fi = lane < k ? si2[lane] : INT_MAX;
    }
    // softmax over the k selected scores
    if (lane >= k) { fv = -INFINITY; fi = INT_MAX; }
    const float m = key2f(__reduce_max_sync(0xffffffffu, f2key(fv)));
    float e = lane < k ? expf(fv - m) : 0.f;
    float zsum = e;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) zsum += __shfl_xor_sync(0xffffffffu, zsum, off);
    // ascending slot order: bitonic network across the 32 lanes
    int key = fi;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const int pk = __shfl_xor_sync(0xffffffffu, key, stride);
            const float pe = __shfl_xor_sync(0xffffffffu, e, stride);
            const bool up = (lane & size) == 0;
            const bool lower = (lane & stride) == 0;
            const bool take_min = (up == lower);
            const bool mine = take_min ? (key <= pk) : (key >= pk);
            key = mine ? key : pk;
            e = mine ? e : pe;
        }
    }
    if (lane < k) {
        const int64_t tokoff = ((b * a.H + h) * a.T + t) * k;     // [B, H, T, k] layout
        a.idx[side][tokoff + lane] = key;
        a.w[side][tokoff + lane] = e / zsum;
    }
}
// ------------------------------------------------------------------------------------------
// Kernel B, wide lists (k > 32): insertion-based merge and candidate selection
// ------------------------------------------------------------------------------------------
template <class D, int L>
__global__ void __launch_bounds__(F_THREADS) k_addr_finalize_wide(const AddrArgs a) {
    extern __shared__ __align__(16) float smB[];
    const int tid = threadIdx.x;
    float* A1v = smB + tid;                       // exact top-k of half 1 (fp32 value, column), pitch F_THREADS
    int* A1i = reinterpret_cast<int*>(smB + 1 * L * F_THREADS) + tid;
    float* A2v = smB + 2 * L * F_THREADS + tid;   // exact top-k of half 2
    int* A2i = reinterpret_cast<int*>(smB + 3 * L * F_THREADS) + tid;
    float* Fv = smB + 4 * L * F_THREADS + tid;    // final selection (fp32 score, slot)
    int* Fi = reinterpret_cast<int*>(smB + 5 * L * F_THREADS) + tid;

    const int side = blockIdx.y / a.H, h = blockIdx.y % a.H;
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    const int64_t u = static_cast<int64_t>(blockIdx.x) * F_THREADS + tid;
    if (u >= BT) return;   // no block-level synchronisation below
    const int k = a.kk[side];
    const int S = a.S;
    const int64_t b = u / a.T, t = u - b * a.T;
    TokenCtx c;
    c.err = a.err;
    c.P = a.P[side];
    c.X = a.X[side];
    c.xoff = ((b * a.H + h) * a.T + t) * a.dk;
    c.prow0 = static_cast<int64_t>(h) * 2 * S;
    c.dk = a.dk;
    c.S = S;

    double eps = 0.0;
    if (c.P != nullptr) {
        float ss = 0.f;
        for (int d = 0; d < a.dk; ++d) {
            const float xv = load_elem<D>(c.X, c.xoff + d);
            ss = fmaf(xv, xv, ss);
        }
        eps = static_cast<double>(a.cbound) * static_cast<double>(a.pnorm[side * a.H + h]) *
              static_cast<double>(sqrtf(ss)) * (1.0 + 0x1p-12);
    }

    float amax[2];
#pragma unroll 1
    for (int hf = 0; hf < 2; ++hf) {
        TopList<L> top;
        top.clear();
        for (int cc = 0; cc < a.ncc; ++cc) {
            const int64_t base = part_at(blockIdx.y, a.ncc, hf * a.ncc + cc, BT, u, L, 0);
            for (int p = 0; p < L; ++p) {
                const float v = a.part_v[base + p];
                const int i = a.part_i[base + p];
                if (!top.admits(v, i)) break;
                top.push(v, i);
            }
        }
        float* Av = hf ? A2v : A1v;
        int* Ai = hf ? A2i : A1i;
        bool certified = (S <= k);
        if (!certified) certified = static_cast<double>(pick(top.v, k - 1)) - static_cast<double>(pick(top.v, k)) > 2.0 * eps;
        if (certified) {
#pragma unroll
            for (int p = 0; p < L; ++p)
                if (p < k) { Av[p * F_THREADS] = top.v[p]; Ai[p * F_THREADS] = top.i[p]; }
        } else {
            float lv[L];
            int li[L];
#pragma unroll
            for (int p = 0; p < L; ++p) { lv[p] = top.v[p]; li[p] = top.i[p]; }
            stat_add(c.err, STAT_HALF_BAND);
            resolve_half<D, L>(lv, li, k, eps, c, hf, Av, Ai, F_THREADS);
        }
        amax[hf] = fmaxf(fabsf(Av[0]), fabsf(Av[(k - 1) * F_THREADS]));
    }

    // Candidates of the outer sum.  theta = a provable lower bound on the k-th best fp32 sum:
    // the first a entries of T1 times the first ceil(k/a) of T2 give >= k sums >= it.
    const double epsc = 2.0 * eps + 0x1p-22 * (static_cast<double>(amax[0]) + static_cast<double>(amax[1]));
    float theta = -INFINITY;
    for (int aa = 1;; aa *= 2) {
        if (aa > k) aa = k;
        const int bb = (k + aa - 1) / aa;
        theta = fmaxf(theta, A1v[(aa - 1) * F_THREADS] + A2v[(bb - 1) * F_THREADS]);
        if (aa == k) break;
    }
    const float lo = __double2float_rd(static_cast<double>(theta) - 2.0 * epsc);
    TopList<L> cand;
    cand.clear();
    for (int p1 = 0; p1 < k; ++p1) {
        const float a1 = A1v[p1 * F_THREADS];
        const int i1 = A1i[p1 * F_THREADS];
        if (a1 + A2v[0] < lo) break;
        for (int p2 = 0; p2 < k; ++p2) {
            const float cs = a1 + A2v[p2 * F_THREADS];
            if (cs < lo) break;
            const int f = i1 * S + A2i[p2 * F_THREADS];
            if (cand.admits(cs, f)) cand.push(cs, f);
        }
    }
    bool certified = (k == 1);
    if (!certified) certified = static_cast<double>(pick(cand.v, k - 1)) - static_cast<double>(pick(cand.v, k)) > 2.0 * epsc;
    if (certified) {
#pragma unroll
        for (int p = 0; p < L; ++p)
            if (p < k) { Fv[p * F_THREADS] = cand.v[p]; Fi[p * F_THREADS] = cand.i[p]; }
    } else {
        float cv[L];
        int cf[L];
#pragma unroll
        for (int p = 0; p < L; ++p) { cv[p] = cand.v[p]; cf[p] = cand.i[p]; }
        stat_add(c.err, STAT_COMB_BAND);
        resolve_combined<D, L>(cv, cf, k, epsc, c, A1v, A1i, A2v, A2i, Fv, Fi, F_THREADS);
    }

    // softmax over the selected scores, then ascending slot order
    float m = -INFINITY;
    for (int p = 0; p < k; ++p) m = fmaxf(m, Fv[p * F_THREADS]);
    float z = 0.f;
    for (int p = 0; p < k; ++p) {
        const float e = expf(Fv[p * F_THREADS] - m);
        Fv[p * F_THREADS] = e;
        z += e;
    }
    const float rz = 1.f / z;
    const int64_t tokoff = ((b * a.H + h) * a.T + t) * k;     // [B, H, T, k] layout
    int32_t* oi = a.idx[side] + tokoff;
    float* ow = a.w[side] + tokoff;
    // selection sort by slot (k <= 64; slots are distinct)
    int last = -1;
    for (int r = 0; r < k; ++r) {
        int best = INT_MAX, bp = 0;
        for (int p = 0; p < k; ++p) {
            const int f = Fi[p * F_THREADS];
            if (f > last && f < best) { best = f; bp = p; }
        }
        oi[r] = best;
        ow[r] = Fv[bp * F_THREADS] * rz;
        last = best;
    }
}

// ------------------------------------------------------------------------------------------
// max_j ||P_j|| per (side, head)
// ------------------------------------------------------------------------------------------
template <class D>
__global__ void __launch_bounds__(256) k_pnorm(const AddrArgs a) {
    const int side = blockIdx.x / a.H, h = blockIdx.x % a.H;
    const void* P = a.P[side];
    __shared__ float red[256];
    float mx = 0.f;
    for (int j = threadIdx.x; j < 2 * a.S; j += 256) {
        const int64_t row = (static_cast<int64_t>(h) * 2 * a.S + j) * a.dk;
        float ss = 0.f;
        for (int d = 0; d < a.dk; ++d) {
            const float p = load_elem<D>(P, row + d);
            ss = fmaf(p, p, ss);
        }
        mx = fmaxf(mx, sqrtf(ss));
    }
    red[threadIdx.x] = mx;
    __syncthreads();
    for (int s = 128; s > 0; s >>= 1) {
        if (threadIdx.x < s) red[threadIdx.x] = fmaxf(red[threadIdx.x], red[threadIdx.x + s]);
        __syncthreads();
    }
    if (threadIdx.x == 0) a.pnorm[blockIdx.x] = red[0] * (1.f + 0x1p-12f);
}

// ------------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------------
AddrPlan addr_plan(int dtype, int direct, int B, int H, int T, int dk, int S, int kmax) {
    AddrPlan p;
    p.L = (kmax <= 8 ? 8 : kmax <= 16 ? 16 : kmax <= 32 ? 32 : 64) + 4;
    p.mma = mma_path_supported(dtype, direct, dk, S, kmax);
    const int64_t tiles = (static_cast<int64_t>(B) * T + A_TOK - 1) / A_TOK;
    const int64_t base = 2LL * H * tiles * 2;   // sides x heads x token tiles x halves
    int ncc = 1;
    while ((S + ncc - 1) / ncc > 512) ncc *= 2;                      // chunks of <= 512 columns
    while (base * ncc < 512 && (S / (2 * ncc)) >= 64) ncc *= 2;      // enough CTAs, chunks >= 64 columns
    p.ncc = ncc;
    p.cw = (S + ncc - 1) / ncc;
    return p;
}

size_t addr_partial_bytes(const AddrPlan& plan, int B, int H, int T) {
    return static_cast<size_t>(2) * H * (2 * plan.ncc) * plan.L * static_cast<size_t>(B) * T * (sizeof(float) + sizeof(int));
}

template <class D, int L>
static cudaError_t launch_finalize(const AddrArgs& a, cudaStream_t stream) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    dim3 gB(static_cast<unsigned>((BT + F_THREADS - 1) / F_THREADS), 2 * a.H);
    cudaError_t e;
    if constexpr (L <= 36) {
        dim3 gW(static_cast<unsigned>((BT + FW_WARPS - 1) / FW_WARPS), 2 * a.H);
        k_addr_finalize<D, L><<<gW, FW_WARPS * 32, 0, stream>>>(a);
    } else {
        const size_t smB = static_cast<size_t>(6) * L * F_THREADS * sizeof(float);
        e = cudaFuncSetAttribute(k_addr_finalize_wide<D, L>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smB));
        if (e != cudaSuccess) return e;
        k_addr_finalize_wide<D, L><<<gB, F_THREADS, smB, stream>>>(a);
    }
    return cudaGetLastError();
}

template <class D, int L>
static cudaError_t launch_typed(const AddrPlan& plan, const AddrArgs& a, cudaStream_t stream) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    if (a.P[0] != nullptr) {
        k_pnorm<D><<<2 * a.H, 256, 0, stream>>>(a);
    }
    if (plan.mma) {
        cudaError_t e = launch_address_mma(plan, a, stream);
        if (e != cudaSuccess) return e;
        return launch_finalize<D, L>(a, stream);
    }
    const size_t smA = (static_cast<size_t>(a.dk) * A_TOK + (a.P[0] ? static_cast<size_t>(a.dk) * A_PPITCH : 0)) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k_addr_scores<D, L>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smA));
    if (e != cudaSuccess) return e;
    dim3 gA(static_cast<unsigned>((BT + A_TOK - 1) / A_TOK), 2 * plan.ncc, 2 * a.H);
    k_addr_scores<D, L><<<gA, A_TOK, smA, stream>>>(a);
    return launch_finalize<D, L>(a, stream);
}

template <class D>
static cudaError_t launch_dtype(const AddrPlan& plan, const AddrArgs& a, cudaStream_t stream) {
    switch (plan.L) {
        case 12: return launch_typed<D, 12>(plan, a, stream);
        case 20: return launch_typed<D, 20>(plan, a, stream);
        case 36: return launch_typed<D, 36>(plan, a, stream);
        case 68: return launch_typed<D, 68>(plan, a, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_address(int dtype, const AddrPlan& plan, const AddrArgs& a, cudaStream_t stream) {
    return dtype == 0 ? launch_dtype<F32>(plan, a, stream) : launch_dtype<BF16>(plan, a, stream);
}

}  // namespace sdm
