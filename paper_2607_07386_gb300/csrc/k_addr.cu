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
    unsigned* stat;     // per-warp event counters in shared memory (nullptr: count in err directly)
    bool count_band;    // count band events (false when an earlier pass counted them)
    const void* P;      // P of this side (nullptr = DIRECT)
    const void* X;
    int64_t xoff;       // element offset of the token's x row
    int64_t prow0;      // row of P for column 0 of half 0 (= h * 2S)
    int dk, S;
};

// Event counter (called by one lane): per-warp shared counters, flushed once per warp,
// keep the diagnostics off the global atomic unit.
__device__ __forceinline__ void tstat(const TokenCtx& c, int which, unsigned n = 1u) {
    if (c.stat) c.stat[which] += n;
    else stat_add(c.err, which, n);
}

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
        if (best < 0) {                 // list not sorted by value: never for the lists built here
            flag_error(c.err, ERR_SELECT);
            chosen[r] = -1;
            continue;
        }
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
        if (best < 0) {
            Av[(cin + r) * pitch] = -INFINITY;
            Ai[(cin + r) * pitch] = 0;
            continue;
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
        if (best < 0) {                 // candidate list not sorted by value: never here
            flag_error(c.err, ERR_SELECT);
            Fv[r * pitch] = -INFINITY;
            Fi[r * pitch] = 0;
            continue;
        }
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

// All decisions of the warp finalize run in fp32 (GB300's float64 rate is a small
// fraction of its fp32 rate): error bounds are rounded up and differences rounded down
// (directed-rounding intrinsics), so every "certain" decision is also certain in exact
// arithmetic.  float64 remains only in the serial fallbacks.

// Float-float value h + l (|l| <= ulp(h)/2) with an error bound b on its distance to the
// float64 score of the definition.
struct FF {
    float h, l, b;
};

__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
    s = __fadd_rn(a, b);
    const float bp = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bp)), __fsub_rn(b, bp));
}

// Compensated score of column j of half hf, computed by the whole warp (every lane gets
// the result).  Lane l owns the terms d = l + 32 r (its x values are in xr).  Every product
// is split exactly (p + pe = P x; pe = 0 for bf16 operands) and every addition of the main
// sum -- within a lane and across the butterfly -- exactly by TwoSum; only the error terms
// are summed in plain fp32.  With n = d_k terms and u = 2^-24 the result s + e differs
// from the exact dot product by at most 2 n (n + 1) u^2 (1.03) sum|P x| <= 2^-31 sum|P x|
// for n <= 256, whatever the order of the additions.  The float64 sequential sum of the
// definition lies within (n - 1) 2^-53 sum|P x| of the exact value, so b = 2^-28 sum|P x|
// covers the distance to it with margin (also for the rounding of sum|P x| itself).
// DIRECT addressing: the score is x itself, exact.
template <class D>
__device__ FF ff_score_warp(const TokenCtx& c, const float (&xr)[8], int hf, int j, int lane) {
    if (c.P == nullptr) return FF{load_elem<D>(c.X, c.xoff + static_cast<int64_t>(hf) * c.S + j), 0.f, 0.f};
    const int64_t prow = (c.prow0 + static_cast<int64_t>(hf) * c.S + j) * c.dk;
    float pv[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        const int d = lane + 32 * r;
        pv[r] = (r * 32 < c.dk && d < c.dk) ? load_elem<D>(c.P, prow + d) : 0.f;
    }
    float sum = 0.f, err = 0.f, mag = 0.f;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        if (r * 32 < c.dk) {
            const float p = __fmul_rn(pv[r], xr[r]);
            const float pe = __fmaf_rn(pv[r], xr[r], -p);
            float t, e2;
            two_sum(sum, p, t, e2);
            sum = t;
            err = __fadd_rn(err, __fadd_rn(e2, pe));
            mag = __fadd_rn(mag, fabsf(p));
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float so = __shfl_xor_sync(0xffffffffu, sum, off);
        const float eo = __shfl_xor_sync(0xffffffffu, err, off);
        const float mo = __shfl_xor_sync(0xffffffffu, mag, off);
        float t, e2;
        two_sum(sum, so, t, e2);                   // same t and e2 in both lanes of the pair
        sum = t;
        err = __fadd_rn(__fadd_rn(err, eo), e2);   // (err + eo) is the same in both lanes
        mag = __fadd_rn(mag, mo);
    }
    FF r;
    r.h = __fadd_rn(sum, err);                      // FastTwoSum: |err| << |sum|
    r.l = __fsub_rn(err, __fsub_rn(r.h, sum));
    r.b = __fmul_ru(0x1p-28f, mag);
    return r;
}

// a + b for two compensated half scores (the float64 definition adds its two half scores
// with one more rounding of at most 2^-53 of the sum; 2^-44 |sum| covers that and ours).
__device__ __forceinline__ FF ff_add(const FF& a, const FF& b, bool direct) {
    float h, r;
    two_sum(a.h, b.h, h, r);
    const float l = __fadd_rn(__fadd_rn(a.l, b.l), r);
    FF o;
    o.h = __fadd_rn(h, l);
    o.l = __fsub_rn(l, __fsub_rn(o.h, h));
    const float slack = direct ? __fmul_ru(0x1p-52f, fabsf(o.h)) : __fmul_ru(0x1p-44f, fabsf(o.h));
    o.b = __fadd_ru(__fadd_ru(a.b, b.b), slack);
    return o;
}

// Band entries (lane e < m holds entry e: compensated score v, index id) are ranked under
// (score desc, index asc).  Returns false when two entries are closer than their bounds
// (the float64 definition must decide); otherwise the ranks are those of the float64
// definition.  The difference (hf + lf) - (h + l) is formed with TwoSum on the leading
// parts; the roundings of the rest are covered by `slack`.
__device__ __forceinline__ bool rank_band(const FF& v, int id, int m, int lane, int& rank) {
    rank = 0;
    bool unsure = false;
    for (int f = 0; f < m; ++f) {
        const float hf = __shfl_sync(0xffffffffu, v.h, f);
        const float lf = __shfl_sync(0xffffffffu, v.l, f);
        const float bf = __shfl_sync(0xffffffffu, v.b, f);
        const int jf = __shfl_sync(0xffffffffu, id, f);
        if (lane < m && f != lane) {
            float t, r;
            two_sum(hf, -v.h, t, r);
            const float w = __fadd_rn(__fsub_rn(lf, v.l), r);
            const float diff = __fadd_rn(t, w);
            const float slack = __fmul_ru(0x1p-21f, __fadd_ru(__fadd_ru(fabsf(t), fabsf(r)), __fadd_ru(fabsf(lf), fabsf(v.l))));
            const float tol = __fadd_ru(__fadd_ru(bf, v.b), slack);
            if (tol > 0.f && fabsf(diff) <= tol) unsure = true;
            else rank += (diff > 0.f || (diff == 0.f && jf < id)) ? 1 : 0;
        }
    }
    return !__any_sync(0xffffffffu, unsure);
}

// Band of an uncertified top-k boundary in a list of `len` (<= 64) entries sorted by fp32
// value (lane p: entry p in v0/i0, entry p + 32 in v1/i1): entries [cin, cin + m) lie
// within e2 (twice the error bound, rounded up) of the boundary.  False if the band may
// continue past the list or holds more than 32 entries.
__device__ __forceinline__ bool band_of(float v0, float v1, int len, int k, float e2, bool list_is_all, int lane,
                                        int& cin, int& m) {
    const float lo = __fsub_rd(lane_get(v0, v1, k - 1), e2);
    const float hi = __fadd_ru(lane_get(v0, v1, k), e2);
    const float vl = lane_get(v0, v1, len - 1);
    if (!list_is_all && vl != -INFINITY && vl >= lo) return false;
    cin = __popc(__ballot_sync(0xffffffffu, lane < len && v0 > hi)) +
          __popc(__ballot_sync(0xffffffffu, lane + 32 < len && v1 > hi));
    m = __popc(__ballot_sync(0xffffffffu, lane < len && v0 >= lo && v0 <= hi)) +
        __popc(__ballot_sync(0xffffffffu, lane + 32 < len && v1 >= lo && v1 <= hi));
    return m <= 32;
}

// Writes the certain entries [0, cin) and the chosen band entries (in list order) to ov/oi.
__device__ __forceinline__ void emit_band(float v0, int i0, float bv, int bi, bool chosen, int cin, float* ov, int* oi,
                                          int lane) {
    const unsigned ch = __ballot_sync(0xffffffffu, chosen);
    __syncwarp();
    if (lane < cin) { ov[lane] = v0; oi[lane] = i0; }
    if (chosen) {
        const int q = cin + __popc(ch & ((1u << lane) - 1u));
        ov[q] = bv;
        oi[q] = bi;
    }
    __syncwarp();
}

// Warp-cooperative resolution of an uncertified half boundary (e2 = twice the fp32 error
// bound of the scores).  On success writes the exact top-k, in fp32-list order, to
// ov/oi[0, k) and returns true; false when the serial float64 path must decide (band past
// the list, more than 32 band entries, or a near-tie).
enum : int { BAND_DONE = 0, BAND_NEAR_TIE = 1, BAND_OUTSIDE = 2 };

// x[lane + 32 r] of the token (projected mode) for the warp-cooperative rescoring
template <class D>
__device__ __forceinline__ void load_xr(const TokenCtx& c, int lane, float (&xr)[8]) {
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        const int d = lane + 32 * r;
        xr[r] = (c.P != nullptr && r * 32 < c.dk && d < c.dk) ? load_elem<D>(c.X, c.xoff + d) : 0.f;
    }
}

// Band resolvers.  The common-path kernel (MODE 0) does not contain them.
template <class D, int L>
__device__ __forceinline__ int warp_band_half(float v0, int i0, float v1, int i1, int k, float e2, const TokenCtx& c,
                                           int hf, float* ov, int* oi, int lane) {
    float xr[8];
    load_xr<D>(c, lane, xr);
    int cin, m;
    if (!band_of(v0, v1, L, k, e2, c.S <= L, lane, cin, m)) return BAND_OUTSIDE;
    if (lane == 0 && c.count_band) tstat(c, STAT_HALF_BAND_ENTRIES, static_cast<unsigned>(m));
    const int p = min(cin + lane, L - 1);
    const float bv = lane_get(v0, v1, p);
    const int bi = lane_geti(i0, i1, p);
    FF mine{0.f, 0.f, 0.f};
    for (int e = 0; e < m; ++e) {
        const FF sc = ff_score_warp<D>(c, xr, hf, __shfl_sync(0xffffffffu, bi, e), lane);
        if (lane == e) mine = sc;
    }
    int rank;
    if (!rank_band(mine, bi, m, lane, rank)) return BAND_NEAR_TIE;
    emit_band(v0, i0, bv, bi, lane < m && rank < k - cin, cin, ov, oi, lane);
    return BAND_DONE;
}

// Near-tie in the band: float64 scores of the definition (sequential d order, so equal to
// it bit for bit), one lane per band entry; the ranking is then exact.
template <class D>
__device__ __noinline__ void warp_band64(float v0, int i0, float v1, int i1, int len, int k, float e2, bool all,
                                         bool comb, const TokenCtx& c, int hf, float* ov, int* oi, int lane) {
    int cin, m;
    band_of(v0, v1, len, k, e2, all, lane, cin, m);       // succeeded before with the same arguments
    const int p = min(cin + lane, len - 1);
    const float bv = lane_get(v0, v1, p);
    const int bi = lane_geti(i0, i1, p);
    double s64 = 0.0;
    if (lane < m) s64 = comb ? score64<D>(c, 0, bi / c.S) + score64<D>(c, 1, bi % c.S) : score64<D>(c, hf, bi);
    int rank = 0;
    for (int f = 0; f < m; ++f) {
        const double sf = __shfl_sync(0xffffffffu, s64, f);
        const int jf = __shfl_sync(0xffffffffu, bi, f);
        if (lane < m && f != lane && beats64(sf, jf, s64, bi)) ++rank;
    }
    emit_band(v0, i0, bv, bi, lane < m && rank < k - cin, cin, ov, oi, lane);
}

// Descending bitonic sort of 64 floats held two per lane (element lane in a, lane + 32 in b).
__device__ __forceinline__ void warp_sort64_desc(float& a, float& b, int lane) {
#pragma unroll
    for (int size = 2; size <= 64; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            if (stride == 32) {                                 // elements lane and lane + 32
                const float hi = fmaxf(a, b), lo = fminf(a, b);
                a = hi; b = lo;                                 // size == 64: descending
            } else {
                const float pa = __shfl_xor_sync(0xffffffffu, a, stride);
                const float pb = __shfl_xor_sync(0xffffffffu, b, stride);
                const bool lower = (lane & stride) == 0;
                // element e = lane (+ 32): its block of `size` sorts descending iff (e & size) == 0
                const bool desc_a = (lane & size) == 0;
                const bool desc_b = ((lane + 32) & size) == 0;
                a = (lower == desc_a) ? fmaxf(a, pa) : fminf(a, pa);
                b = (lower == desc_b) ? fmaxf(b, pb) : fminf(b, pb);
            }
        }
    }
}

// Compensated score of column j of half hf by one thread (16-byte loads when aligned); the
// same error-free splitting and the same 2^-28 sum|P x| bound as ff_score_warp.
template <class D>
__device__ FF ff_score_thread(const void* P, const void* X, int64_t xoff, int64_t prow0, int dk, int S, int hf, int j) {
    if (P == nullptr) return FF{load_elem<D>(X, xoff + static_cast<int64_t>(hf) * S + j), 0.f, 0.f};
    const int64_t prow = (prow0 + static_cast<int64_t>(hf) * S + j) * dk;
    float sum = 0.f, err = 0.f, mag = 0.f;
    auto term = [&](float pv, float xv) {
        const float p = __fmul_rn(pv, xv);
        const float pe = __fmaf_rn(pv, xv, -p);
        float t, e2;
        two_sum(sum, p, t, e2);
        sum = t;
        err = __fadd_rn(err, __fadd_rn(e2, pe));
        mag = __fadd_rn(mag, fabsf(p));
    };
    const char* pr = static_cast<const char*>(P) + prow * D::BYTES;
    const char* xr = static_cast<const char*>(X) + xoff * D::BYTES;
    if (((reinterpret_cast<uintptr_t>(pr) | reinterpret_cast<uintptr_t>(xr)) & 15) == 0 && (dk * D::BYTES) % 16 == 0) {
        const int nq = dk * D::BYTES / 16;
        for (int q0 = 0; q0 < nq; q0 += 4) {            // four 16-byte loads in flight per operand
            uint4 pq[4], xq[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (q0 + u < nq) {
                    pq[u] = __ldg(reinterpret_cast<const uint4*>(pr) + q0 + u);
                    xq[u] = __ldg(reinterpret_cast<const uint4*>(xr) + q0 + u);
                }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (q0 + u < nq) {
                    float fp[D::E], fx[D::E];
                    unpack16<D>(pq[u], fp);
                    unpack16<D>(xq[u], fx);
#pragma unroll
                    for (int e = 0; e < D::E; ++e) term(fp[e], fx[e]);
                }
        }
    } else {
        for (int d = 0; d < dk; ++d) term(load_elem<D>(P, prow + d), load_elem<D>(X, xoff + d));
    }
    FF r;
    r.h = __fadd_rn(sum, err);
    r.l = __fsub_rn(err, __fsub_rn(r.h, sum));
    r.b = __fmul_ru(0x1p-28f, mag);
    return r;
}

// The band of a half boundary reaches past the kept list: exact top-k over the whole half,
// one column per lane at a time.
//   pass 1: fp32 scores (sequential FMA, error <= eps), each lane keeps the top 2 of its
//           columns j = lane (mod 32); theta = k-th largest of those 64 values (>= k columns
//           reach it, so the k-th largest exact score is >= theta - eps);
//   pass 2: columns with fp32 score >= theta - 2 eps (a superset of the exact top-k) are
//           collected (at most 64, else false), rescored compensated and ranked.
// Writes the top-k in order (value fl32 of the compensated score, index) to ov/oi.
template <class D>
__device__ __noinline__ bool warp_full_half(int k, float e2, const TokenCtx& c, int hf, float* ov, int* oi,
                                            int* scratch, int lane) {
    const int S = c.S;
    const char* xr = static_cast<const char*>(c.X) + c.xoff * D::BYTES;
    const bool vec = ((reinterpret_cast<uintptr_t>(c.P) | reinterpret_cast<uintptr_t>(xr)) & 15) == 0 &&
                     (c.dk * D::BYTES) % 16 == 0;
    auto fp32_score = [&](int j) -> float {             // sequential FMA over d (error <= eps)
        const int64_t prow = (c.prow0 + static_cast<int64_t>(hf) * S + j) * c.dk;
        float acc = 0.f;
        if (vec) {
            const uint4* pr = reinterpret_cast<const uint4*>(static_cast<const char*>(c.P) + prow * D::BYTES);
            for (int q = 0; q < c.dk * D::BYTES / 16; ++q) {
                float fp[D::E], fx[D::E];
                unpack16<D>(__ldg(pr + q), fp);
                unpack16<D>(__ldg(reinterpret_cast<const uint4*>(xr) + q), fx);
#pragma unroll
                for (int e = 0; e < D::E; ++e) acc = fmaf(fp[e], fx[e], acc);
            }
        } else {
            for (int d = 0; d < c.dk; ++d) acc = fmaf(load_elem<D>(c.P, prow + d), load_elem<D>(c.X, c.xoff + d), acc);
        }
        return acc;
    };
    float t1 = -INFINITY, t2 = -INFINITY;
    for (int j0 = 0; j0 < S; j0 += 32) {
        const int j = j0 + lane;
        const float sc = j < S ? fp32_score(j) : -INFINITY;
        t2 = fmaxf(t2, fminf(t1, sc));
        t1 = fmaxf(t1, sc);
    }
    warp_sort64_desc(t1, t2, lane);
    const float theta = lane_get(t1, t2, k - 1);
    const float lo = __fsub_rd(theta, e2);
    int m = 0;
    for (int j0 = 0; j0 < S; j0 += 32) {
        const int j = j0 + lane;
        const bool keep = j < S && fp32_score(j) >= lo;
        const unsigned mask = __ballot_sync(0xffffffffu, keep);
        const int pos = m + __popc(mask & ((1u << lane) - 1u));
        if (keep && pos < 64) scratch[pos] = j;
        m += __popc(mask);
    }
    if (m > 64) return false;
    __syncwarp();
    const int j0 = lane < m ? scratch[lane] : 0;
    const int j1 = lane + 32 < m ? scratch[lane + 32] : 0;
    __syncwarp();
    FF f0{0.f, 0.f, 0.f}, f1{0.f, 0.f, 0.f};
    if (lane < m) f0 = ff_score_thread<D>(c.P, c.X, c.xoff, c.prow0, c.dk, S, hf, j0);
    if (lane + 32 < m) f1 = ff_score_thread<D>(c.P, c.X, c.xoff, c.prow0, c.dk, S, hf, j1);
    // rank both own entries against all m (pairs closer than their bounds: give up)
    int r0 = 0, r1 = 0;
    bool unsure = false;
    for (int f = 0; f < m; ++f) {
        const int src = f & 31;
        const bool hi = f >= 32;
        const float hA = __shfl_sync(0xffffffffu, f0.h, src), hB = __shfl_sync(0xffffffffu, f1.h, src);
        const float lA = __shfl_sync(0xffffffffu, f0.l, src), lB = __shfl_sync(0xffffffffu, f1.l, src);
        const float bA = __shfl_sync(0xffffffffu, f0.b, src), bB = __shfl_sync(0xffffffffu, f1.b, src);
        const FF ff{hi ? hB : hA, hi ? lB : lA, hi ? bB : bA};
        const int jf = lane_geti(j0, j1, f);
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int e = lane + 32 * q;
            const FF& mine = q ? f1 : f0;
            const int je = q ? j1 : j0;
            if (e < m && e != f) {
                float t, r;
                two_sum(ff.h, -mine.h, t, r);
                const float w = __fadd_rn(__fsub_rn(ff.l, mine.l), r);
                const float diff = __fadd_rn(t, w);
                const float slack = __fmul_ru(0x1p-21f, __fadd_ru(__fadd_ru(fabsf(t), fabsf(r)), __fadd_ru(fabsf(ff.l), fabsf(mine.l))));
                const float tol = __fadd_ru(__fadd_ru(ff.b, mine.b), slack);
                if (tol > 0.f && fabsf(diff) <= tol) unsure = true;
                else if (diff > 0.f || (diff == 0.f && jf < je)) { if (q) ++r1; else ++r0; }
            }
        }
    }
    if (__any_sync(0xffffffffu, unsure)) return false;
    __syncwarp();
    if (lane < m && r0 < k) { ov[r0] = f0.h; oi[r0] = j0; }
    if (lane + 32 < m && r1 < k) { ov[r1] = f1.h; oi[r1] = j1; }
    __syncwarp();
    return true;
}

// Same for the outer-sum boundary over a candidate list of `len` (<= 64) entries: slot
// f = i S + j is rescored as the sum of the compensated half scores of column i (half 0)
// and column j (half 1).
template <class D>
__device__ __forceinline__ int warp_band_comb(float v0, int f0, float v1, int f1, int len, int k, float e2c,
                                           const TokenCtx& c, bool all, float* ov, int* oi, int lane) {
    float xr[8];
    load_xr<D>(c, lane, xr);
    int cin, m;
    if (!band_of(v0, v1, len, k, e2c, all, lane, cin, m)) return BAND_OUTSIDE;
    if (lane == 0 && c.count_band) tstat(c, STAT_COMB_BAND_ENTRIES, static_cast<unsigned>(m));
    const int p = min(cin + lane, len - 1);
    const float bv = lane_get(v0, v1, p);
    const int bf = lane_geti(f0, f1, p);
    FF mine{0.f, 0.f, 0.f};
    for (int e = 0; e < m; ++e) {
        const int fe = __shfl_sync(0xffffffffu, bf, e);
        const FF s1 = ff_score_warp<D>(c, xr, 0, fe / c.S, lane);
        const FF s2 = ff_score_warp<D>(c, xr, 1, fe % c.S, lane);
        const FF sum = ff_add(s1, s2, c.P == nullptr);
        if (lane == e) mine = sum;
    }
    int rank;
    if (!rank_band(mine, bf, m, lane, rank)) return BAND_NEAR_TIE;
    emit_band(v0, f0, bv, bf, lane < m && rank < k - cin, cin, ov, oi, lane);
    return BAND_DONE;
}

// Three passes over token-sides, each kernel holding only the code its cases need (the
// band code's registers and instruction footprint would otherwise slow the common path):
//   MODE 0: every token-side; those whose two half boundaries and outer-sum boundary are
//           all certified are finished, the others go to queue A (nothing written);
//   MODE 1: queue A, with band resolution by compensated rescoring; near-ties and bands
//           that leave the kept lists go to queue B;
//   MODE 2: queue B (or every token-side when there is no queue) with every path.
enum : int { FIN_FAST = 0, FIN_BAND = 1, FIN_FULL = 2 };

template <class D, int L, int MODE>
__global__ void __launch_bounds__(FW_WARPS * 32, 4) k_addr_finalize(const AddrArgs a) {
    static_assert(L <= 36, "warp finalize handles k <= 32");
    __shared__ float wv[FW_WARPS][3][64];
    __shared__ int wi[FW_WARPS][3][64];
    __shared__ unsigned wstat[FW_WARPS][STAT_COUNT];
    const int lane = threadIdx.x & 31, wq = threadIdx.x >> 5;
    if (lane < STAT_COUNT) wstat[wq][lane] = 0u;
    __syncwarp();
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    const int64_t all = 2 * a.H * BT;
    const bool queued = a.queue != nullptr;               // then all < 2^31
    int* const qa = queued ? a.queue + 2 : nullptr;        // queue A items
    int* const qb = queued ? a.queue + 2 + all : nullptr;  // queue B items
    const int64_t items = MODE == FIN_FAST || !queued ? all
                        : static_cast<int64_t>(reinterpret_cast<volatile int*>(a.queue)[MODE == FIN_BAND ? 0 : 1]);
    // persistent warps: a warp takes token-sides it, it + (all warps), ...
    for (int64_t it = static_cast<int64_t>(blockIdx.x) * FW_WARPS + wq; it < items;
         it += static_cast<int64_t>(gridDim.x) * FW_WARPS) {
    int64_t item, u, b, t;
    int z;
    if (queued) {                                          // 32-bit index arithmetic
        const uint32_t it32 = MODE == FIN_FAST ? static_cast<uint32_t>(it)
                            : static_cast<uint32_t>((MODE == FIN_BAND ? qa : qb)[it]);
        const uint32_t z32 = it32 / static_cast<uint32_t>(BT);
        const uint32_t u32 = it32 - z32 * static_cast<uint32_t>(BT);
        const uint32_t b32 = u32 / static_cast<uint32_t>(a.T);
        item = it32; z = static_cast<int>(z32); u = u32; b = b32; t = u32 - b32 * static_cast<uint32_t>(a.T);
    } else {
        item = it;
        z = static_cast<int>(item / BT);
        u = item - z * BT;
        b = u / a.T;
        t = u - b * a.T;
    }
    const int side = z / a.H, h = z % a.H;
    const int k = a.kk[side];
    const int S = a.S;
    TokenCtx c;
    c.err = a.err;
    c.stat = wstat[wq];
    c.count_band = MODE != FIN_FULL || !queued;
    c.P = a.P[side];
    c.X = a.X[side];
    c.xoff = ((b * a.H + h) * a.T + t) * a.dk;
    c.prow0 = static_cast<int64_t>(h) * 2 * S;
    c.dk = a.dk;
    c.S = S;
    float* sv0 = wv[wq][0]; int* si0 = wi[wq][0];          // staging / merge output / A1
    float* sv1 = wv[wq][1]; int* si1 = wi[wq][1];          // A2
    float* sv2 = wv[wq][2]; int* si2 = wi[wq][2];          // candidates / final

    float e2 = 0.f;                                        // 2 x the fp32 score error bound, rounded up
    if (c.P != nullptr) {
        float ss = 0.f;
        for (int d = lane; d < a.dk; d += 32) {
            const float xv = load_elem<D>(c.X, c.xoff + d);
            ss = fmaf(xv, xv, ss);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        // (1 + 2^-12) covers the roundings of ||x||^2, its square root and the products
        e2 = __fmul_ru(__fmul_ru(__fmul_ru(2.f * a.cbound, a.pnorm[side * a.H + h]), sqrtf(ss)), 1.f + 0x1p-12f);
    }
    const double eps = 0.5 * static_cast<double>(e2);    // for the serial float64 fallbacks

    float av[2], bv[2];      // A1 and A2 after certification: lane p holds entry p (p < k)
    int ai[2], bi[2];
    float amax[2];
    bool deferred = false;
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
            certified = __fsub_rd(vk, vk1) > e2;
        }
        if (MODE == FIN_FAST && !certified) {
            deferred = true;
            break;
        }
        if (!certified) {
            if (lane == 0 && c.count_band) tstat(c, STAT_HALF_BAND);
            const int res = warp_band_half<D, L>(v0, i0, v1, i1, k, e2, c, hf, sv0, si0, lane);
            bool done = res == BAND_DONE;
            if (MODE == FIN_BAND && !done) {
                deferred = true;
                break;
            }
            if (res == BAND_NEAR_TIE) {
                if (lane == 0) tstat(c, STAT_BAND_F64);
                warp_band64<D>(v0, i0, v1, i1, L, k, e2, S <= L, false, c, hf, sv0, si0, lane);
                done = true;
            } else if (res == BAND_OUTSIDE) {
                if (lane == 0) tstat(c, STAT_HALF_FULL);
                done = c.P != nullptr && warp_full_half<D>(k, e2, c, hf, sv0, si0, si2, lane);
            }
            if (!done) {
                if (lane == 0) tstat(c, STAT_SERIAL);
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
    if (MODE != FIN_FULL && deferred) {
        if (lane == 0) {
            if (MODE == FIN_FAST) qa[atomicAdd(a.queue, 1)] = static_cast<int>(item);
            else qb[atomicAdd(a.queue + 1, 1)] = static_cast<int>(item);
        }
        __syncwarp();
        continue;
    }

    // combined: k-way merge of the rows (lane i: row i; head = A1[i] + A2[j])
    // outer-sum bound: both half errors plus the fp32 rounding of A1 + A2 (rounded up, x2)
    const float e2c = __fadd_ru(__fmul_ru(2.f, e2), __fmul_ru(0x1p-21f, __fadd_ru(amax[0], amax[1])));
    const double epsc = 0.5 * static_cast<double>(e2c);  // for the serial float64 fallback
    int j = 0;
    const float b0v = __shfl_sync(0xffffffffu, bv[0], 0);
    const int b0i = __shfl_sync(0xffffffffu, bi[0], 0);
    float head = lane < k ? av[0] + b0v : -INFINITY;
    int flat = ai[0] * S + b0i;
    float cv0 = -INFINITY, cv1 = -INFINITY;    // candidate r in lane r (r < 32) / lane r-32
    int cf0 = INT_MAX, cf1 = INT_MAX;
    auto merge_steps = [&](int r0, int r1) {
        for (int r = r0; r < r1; ++r) {
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
    };
    merge_steps(0, MODE == FIN_FAST ? k + 1 : L);           // certification needs entries k-1 and k
    bool certified = (k == 1);
    if (!certified) {
        const float ck = lane_get(cv0, cv1, k - 1), ck1 = lane_get(cv0, cv1, k);
        certified = (ck1 == -INFINITY) || (__fsub_rd(ck, ck1) > e2c);
    }
    float fv = cv0;
    int fi = cf0;
    if (MODE == FIN_FAST && !certified) {
        if (lane == 0) qa[atomicAdd(a.queue, 1)] = static_cast<int>(item);
        __syncwarp();
        continue;
    }
    if (!certified) {
        if (lane == 0 && c.count_band) tstat(c, STAT_COMB_BAND);
        // band may continue past the L candidates: extend the merge to 64 (or all k^2)
        int len = L;
        const float vl = lane_get(cv0, cv1, L - 1);
        if (k * k > L && vl != -INFINITY &&
            vl >= __fsub_rd(lane_get(cv0, cv1, k - 1), e2c)) {
            if (lane == 0) tstat(c, STAT_COMB_MERGE);
            len = min(64, k * k);
            merge_steps(L, len);
        }
        const int res = warp_band_comb<D>(cv0, cf0, cv1, cf1, len, k, e2c, c, len >= k * k, sv2, si2, lane);
        if (MODE == FIN_BAND && res != BAND_DONE) {
            if (lane == 0) qb[atomicAdd(a.queue + 1, 1)] = static_cast<int>(item);
            __syncwarp();
            continue;
        }
        if (res == BAND_NEAR_TIE) {
            if (lane == 0) tstat(c, STAT_BAND_F64);
            warp_band64<D>(cv0, cf0, cv1, cf1, len, k, e2c, len >= k * k, true, c, 0, sv2, si2, lane);
        } else if (res == BAND_OUTSIDE) {
            if (lane == 0) { tstat(c, STAT_COMB_FULL); tstat(c, STAT_SERIAL); }
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
    __syncwarp();                                           // per-warp staging is reused
    }
    __syncwarp();
    if (lane > 0 && lane < STAT_COUNT && wstat[wq][lane] != 0u) stat_add(a.err, lane, wstat[wq][lane]);
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
    c.stat = nullptr;
    c.count_band = true;
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
    // one warp per row of P (lanes split d), four consecutive rows per warp; the row norms are
    // folded into pnorm[side * H + h] (zeroed before) by an integer atomicMax, which orders
    // non-negative floats correctly.  (1 + 2^-12) covers the roundings of the norm.
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rows = 2 * a.S;
    const int64_t total = static_cast<int64_t>(2) * a.H * rows;
    const int64_t r0 = (static_cast<int64_t>(blockIdx.x) * 8 + warp) * 4;
    int zcur = -1;
    float mx = 0.f;
    for (int q = 0; q < 4; ++q) {
        const int64_t r = r0 + q;
        if (r >= total) break;                       // warp-uniform
        const int zs = static_cast<int>(r / rows);
        const int64_t jrow = r - static_cast<int64_t>(zs) * rows;
        const int side = zs / a.H, h = zs % a.H;
        const int64_t row = (static_cast<int64_t>(h) * rows + jrow) * a.dk;
        float ss = 0.f;
        for (int d = lane; d < a.dk; d += 32) {
            const float p = load_elem<D>(a.P[side], row + d);
            ss = fmaf(p, p, ss);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        const float nrm = sqrtf(ss) * (1.f + 0x1p-12f);
        if (zs != zcur) {
            if (zcur >= 0 && lane == 0) atomicMax(reinterpret_cast<int*>(a.pnorm) + zcur, __float_as_int(mx));
            zcur = zs;
            mx = 0.f;
        }
        mx = fmaxf(mx, nrm);
    }
    if (zcur >= 0 && lane == 0) atomicMax(reinterpret_cast<int*>(a.pnorm) + zcur, __float_as_int(mx));
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
    // FFMA path: more chunks when the token tiles alone give too few CTAs.  The tensor-core
    // path keeps one chunk per half (512 TMEM columns), so the one-thread passes finish it.
    if (!p.mma)
        while (base * ncc < 512 && (S / (2 * ncc)) >= 64) ncc *= 2;  // enough CTAs, chunks >= 64 columns
    p.ncc = ncc;
    p.cw = (S + ncc - 1) / ncc;
    return p;
}

// Queues of the three-pass warp finalize (0 when the item ids would not fit in int32: a
// single full pass is used then).
size_t addr_queue_bytes(int B, int H, int T) {
    const int64_t items = static_cast<int64_t>(2) * H * B * T;
    if (2 * items >= (static_cast<int64_t>(1) << 31) - 2) return 0;
    return static_cast<size_t>(2 + 2 * items) * sizeof(int);       // two counts, queues A and B
}

size_t addr_partial_bytes(const AddrPlan& plan, int B, int H, int T) {
    return static_cast<size_t>(2) * H * (2 * plan.ncc) * plan.L * static_cast<size_t>(B) * T * (sizeof(float) + sizeof(int));
}

// ------------------------------------------------------------------------------------------
// Certified pass, one thread per token-side (one column chunk per half, k <= 32).  Same
// decisions as the warp pass (MODE 0).  The outer sums A1[i] + A2[j] (i, j < k: only they can
// hold the k largest once both half boundaries are certified) are taken in descending order
// from a frontier held in registers: with both lists descending the taken cells form a
// staircase (row i holds the cells j < m_i, m non-increasing) and the next largest sum is one
// of its outer corners, at most 8 of them while at most 35 cells are taken.  k + 1 steps give
// the k-th and (k+1)-th values; the selected cells are the staircase after k steps.  Exact
// tie order is irrelevant: a certified boundary has a positive gap, so equal values never
// straddle it.  Token-sides with an uncertified boundary go to queue A.
// ------------------------------------------------------------------------------------------
constexpr int FT_THREADS = 64;
constexpr int FT_FRONT = 8;       // frontier cells (outer corners of a staircase of <= 35 cells)

// Shared bytes per thread: the first k + 1 values of each half list (32-bit), the first k list
// indices (16-bit: one column chunk per half, indices < 512) and the staircase row counts
// (bytes, k + 1 of them, padded to a word).
__host__ __device__ constexpr int ft_bytes(int km) { return 2 * 4 * (km + 1) + 2 * 2 * km + ((km + 4) & ~3); }

template <class D, int L>
__global__ void __launch_bounds__(FT_THREADS, 8) k_addr_finalize_thread(const AddrArgs a) {
    constexpr int KM = L - 4;                     // largest k served
    static_assert(KM <= 32, "frontier bound holds for k <= 32");
    extern __shared__ float fts[];
    const int tid = threadIdx.x;
    constexpr int W = FT_THREADS;
    // per-thread columns [element][FT_THREADS]: conflict-free for any element index
    float* const A1v = fts + tid;                                             // [KM + 1]
    float* const A2v = fts + (KM + 1) * W + tid;                              // [KM + 1]
    unsigned short* const h16 = reinterpret_cast<unsigned short*>(fts + 2 * (KM + 1) * W);
    unsigned short* const A1i = h16 + tid;                                    // [KM]
    unsigned short* const A2i = h16 + KM * W + tid;                           // [KM]
    unsigned char* const m8 = reinterpret_cast<unsigned char*>(h16 + 2 * KM * W) + tid;   // [KM + 1]

    const uint32_t BT = static_cast<uint32_t>(a.B) * static_cast<uint32_t>(a.T);
    const uint32_t items = 2u * static_cast<uint32_t>(a.H) * BT;      // < 2^31 (a queue exists)
    const uint32_t item = blockIdx.x * FT_THREADS + tid;
    if (item >= items) return;                    // no barrier in this kernel
    const uint32_t z = item / BT, u = item - z * BT;
    const int side = static_cast<int>(z) / a.H, h = static_cast<int>(z) % a.H;
    const int k = a.kk[side];
    const int S = a.S;
    const uint32_t b = u / static_cast<uint32_t>(a.T), t = u - b * static_cast<uint32_t>(a.T);
    const void* X = a.X[side];
    const int64_t xoff = ((static_cast<int64_t>(b) * a.H + h) * a.T + t) * a.dk;

    float e2 = 0.f;
    if (a.P[side] != nullptr) {
        float ss = 0.f;
        const char* xr = static_cast<const char*>(X) + xoff * D::BYTES;
        if ((reinterpret_cast<uintptr_t>(xr) & 15) == 0 && (a.dk * D::BYTES) % 16 == 0) {
            const int nq = a.dk * D::BYTES / 16;
            for (int q0 = 0; q0 < nq; q0 += 4) {
                uint4 xq[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (q0 + u < nq) xq[u] = __ldg(reinterpret_cast<const uint4*>(xr) + q0 + u);
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (q0 + u < nq) {
                        float f[D::E];
                        unpack16<D>(xq[u], f);
#pragma unroll
                        for (int e = 0; e < D::E; ++e) ss = fmaf(f[e], f[e], ss);
                    }
            }
        } else {
            for (int d = 0; d < a.dk; ++d) {
                const float xv = load_elem<D>(X, xoff + d);
                ss = fmaf(xv, xv, ss);
            }
        }
        // (1 + 2^-12) covers the roundings of ||x||^2, its square root and the products
        e2 = __fmul_ru(__fmul_ru(__fmul_ru(2.f * a.cbound, a.pnorm[side * a.H + h]), sqrtf(ss)), 1.f + 0x1p-12f);
    }
    auto defer = [&]() { a.queue[2 + atomicAdd(a.queue, 1)] = static_cast<int>(item); };

    // the two half lists (chunk 0 of each half), first k + 1 entries
    float amax[2];
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
        const int64_t base = part_at(static_cast<int>(z), 1, hf, BT, u, L, 0);
        const float4* pv = reinterpret_cast<const float4*>(a.part_v + base);
        const int4* pi = reinterpret_cast<const int4*>(a.part_i + base);
        float* Av = hf ? A2v : A1v;
        unsigned short* Ai = hf ? A2i : A1i;
#pragma unroll
        for (int q = 0; q < L / 4; ++q) {
            if (4 * q <= k) {
                const float4 v4 = __ldg(pv + q);
                const int4 i4 = __ldg(pi + q);
                const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
                const int ii[4] = {i4.x, i4.y, i4.z, i4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int p = 4 * q + e;
                    if (p <= k && p <= KM) Av[p * W] = vv[e];
                    if (p < k && p < KM) Ai[p * W] = static_cast<unsigned short>(ii[e]);
                }
            }
        }
        const float vk = Av[(k - 1) * W], vk1 = Av[k * W];
        if (!(S <= k || __fsub_rd(vk, vk1) > e2)) { defer(); return; }
        amax[hf] = fmaxf(fabsf(Av[0]), fabsf(vk));
    }
    const float e2c = __fadd_ru(__fmul_ru(2.f, e2), __fmul_ru(0x1p-21f, __fadd_ru(amax[0], amax[1])));

    // staircase walk: k + 1 steps, each taking the largest frontier cell
#pragma unroll
    for (int i = 0; i <= KM; ++i)
        if (i <= k) m8[i * W] = 0;
    float fv[FT_FRONT];
    int fij[FT_FRONT];                            // i | j << 8
#pragma unroll
    for (int f = 0; f < FT_FRONT; ++f) { fv[f] = -INFINITY; fij[f] = 0; }
    const float vmax = A1v[0] + A2v[0];
    fv[0] = vmax;
    float ck = -INFINITY, ck1 = -INFINITY;
    bool full = false;
    for (int r = 0; r <= k; ++r) {
        float bv = fv[0];
        int bf = 0;
#pragma unroll
        for (int f = 1; f < FT_FRONT; ++f) {
            const bool gt = fv[f] > bv;
            bv = gt ? fv[f] : bv;
            bf = gt ? f : bf;
        }
        if (r == k) { ck1 = bv; break; }
        ck = bv;                                   // the k-th value after the last step
        int bij = 0;
#pragma unroll
        for (int f = 0; f < FT_FRONT; ++f) bij = f == bf ? fij[f] : bij;
        const int i = bij & 255, j = bij >> 8;
        m8[i * W] = static_cast<unsigned char>(j + 1);
        // (i, j + 1) becomes a corner once row i - 1 holds more than j + 1 cells
        const bool right = j + 1 < k && (i == 0 || m8[(i - 1) * W] > j + 1);
        // (i + 1, j) becomes a corner when row i + 1 holds exactly j cells
        const bool down = i + 1 < k && m8[(i + 1) * W] == j;
        const float rv = right ? A1v[i * W] + A2v[(j + 1) * W] : -INFINITY;
        const float dv = down ? A1v[(i + 1) * W] + A2v[j * W] : -INFINITY;
#pragma unroll
        for (int f = 0; f < FT_FRONT; ++f)
            if (f == bf) { fv[f] = rv; fij[f] = i | ((j + 1) << 8); }
        bool placed = !down || dv == -INFINITY;
#pragma unroll
        for (int f = 0; f < FT_FRONT; ++f) {
            const bool here = !placed && fv[f] == -INFINITY;
            fv[f] = here ? dv : fv[f];
            fij[f] = here ? ((i + 1) | (j << 8)) : fij[f];
            placed |= here;
        }
        full |= !placed;
    }
    // (-inf cells are padding past a short half list; they only ever supply the (k+1)-th value)
    if (full || !(__fsub_rd(ck, ck1) > e2c)) { defer(); return; }
    // softmax over the k selected scores (the staircase, row by row), then ascending slot order
    // (bitonic network)
    float ew[KM];
    int sl[KM];
    float zsum = 0.f;
    int ci = 0, cj = 0, mi = m8[0];
#pragma unroll
    for (int r = 0; r < KM; ++r) {
        if (r < k) {
            ew[r] = expf((A1v[ci * W] + A2v[cj * W]) - vmax);
            sl[r] = static_cast<int>(A1i[ci * W]) * S + static_cast<int>(A2i[cj * W]);
            zsum += ew[r];
            if (++cj == mi) { ++ci; cj = 0; mi = m8[ci * W]; }
        } else {
            ew[r] = 0.f;
            sl[r] = INT_MAX;
        }
    }
#pragma unroll
    for (int size = 2; size <= KM; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
            for (int i = 0; i < KM; ++i) {
                const int jx = i ^ stride;
                if (jx > i) {
                    const bool up = (i & size) == 0;
                    const bool sw = up ? (sl[i] > sl[jx]) : (sl[i] < sl[jx]);
                    const int si = sl[i];
                    const float ei = ew[i];
                    sl[i] = sw ? sl[jx] : si;  ew[i] = sw ? ew[jx] : ei;
                    sl[jx] = sw ? si : sl[jx]; ew[jx] = sw ? ei : ew[jx];
                }
            }
    const int64_t tokoff = ((static_cast<int64_t>(b) * a.H + h) * a.T + t) * k;
    int32_t* oi = a.idx[side] + tokoff;
    float* ow = a.w[side] + tokoff;
#pragma unroll
    for (int r = 0; r < KM; ++r)
        if (r < k) { oi[r] = sl[r]; ow[r] = ew[r] / zsum; }
}

// ------------------------------------------------------------------------------------------
// Band pass, one thread per token-side of queue A (one column chunk per half, k <= 32): the
// band of an uncertified boundary (entries within twice the error bound of it) is re-ranked
// by compensated scores, one thread computing each score sequentially.  A band that leaves
// the kept candidates, holds more than 32 entries, or has two entries closer than their
// compensated bounds goes to queue B (float64 and whole-half paths).
// ------------------------------------------------------------------------------------------
constexpr int BT_THREADS = 32;
constexpr int BT_BAND = 8;        // band entries re-ranked here; wider bands go to queue B
// Shared bytes per thread: values, candidates and band scratch as 32-bit words, the half
// lists' column indices and the heap positions as 16-bit (one column chunk per half: < 512).
__host__ __device__ constexpr int bt_bytes(int L) { return 4 * (4 * L + (L - 4) + 4 * BT_BAND) + 2 * (2 * L + (L - 4)); }

// f versus e (compensated values): +1 if f is certainly larger, -1 if certainly smaller, 0 if
// equal with zero bounds (exact values: the caller breaks the tie); sets unsure when the two
// are closer than their bounds.
__device__ __forceinline__ int ff_cmp(const FF& f, const FF& e, bool& unsure) {
    float t, r;
    two_sum(f.h, -e.h, t, r);
    const float w = __fadd_rn(__fsub_rn(f.l, e.l), r);
    const float diff = __fadd_rn(t, w);
    const float slack = __fmul_ru(0x1p-21f, __fadd_ru(__fadd_ru(fabsf(t), fabsf(r)), __fadd_ru(fabsf(f.l), fabsf(e.l))));
    const float tol = __fadd_ru(__fadd_ru(f.b, e.b), slack);
    if (tol > 0.f && fabsf(diff) <= tol) { unsure = true; return 0; }
    return diff > 0.f ? 1 : diff < 0.f ? -1 : 0;
}

template <class D, int L>
__global__ void __launch_bounds__(BT_THREADS) k_addr_band_thread(const AddrArgs a) {
    constexpr int KM = L - 4;
    constexpr int LOG = KM <= 8 ? 3 : KM <= 16 ? 4 : 5;
    constexpr int W = BT_THREADS;
    extern __shared__ float bts[];
    const int tid = threadIdx.x;
    float* const A1v = bts + tid;                                              // [L]
    float* const A2v = bts + L * W + tid;                                      // [L]
    float* const hv = bts + 2 * L * W + tid;                                   // [KM]
    float* const ov = bts + (2 * L + KM) * W + tid;                            // [L] candidates
    int* const os = reinterpret_cast<int*>(bts) + (3 * L + KM) * W + tid;      // [L]
    float* const bh = bts + (4 * L + KM) * W + tid;                            // [BT_BAND] band: h
    float* const bl = bts + (4 * L + KM + BT_BAND) * W + tid;                  //                 l
    float* const bb = bts + (4 * L + KM + 2 * BT_BAND) * W + tid;              //                 bound
    int* const bc = reinterpret_cast<int*>(bts) + (4 * L + KM + 3 * BT_BAND) * W + tid;   // chosen
    unsigned short* const h16 = reinterpret_cast<unsigned short*>(bts + (4 * L + KM + 4 * BT_BAND) * W);
    unsigned short* const A1i = h16 + tid;                                     // [L]
    unsigned short* const A2i = h16 + L * W + tid;                             // [L]
    unsigned short* const hp = h16 + 2 * L * W + tid;                          // [KM] row | col << 8

    const uint32_t BT = static_cast<uint32_t>(a.B) * static_cast<uint32_t>(a.T);
    const uint32_t nq = static_cast<uint32_t>(*reinterpret_cast<volatile int*>(a.queue));
    const uint32_t all = 2u * static_cast<uint32_t>(a.H) * BT;
    uint32_t stat_hb = 0, stat_he = 0, stat_cb = 0, stat_ce = 0;
    // grid-stride over queue A (the grid is sized to the SMs, not to the longest queue)
    for (uint32_t q = blockIdx.x * BT_THREADS + tid; q < nq; q += gridDim.x * BT_THREADS) {
        const uint32_t item = static_cast<uint32_t>(a.queue[2 + q]);
        int* const qb = a.queue + 2 + all;
        auto defer = [&]() { qb[atomicAdd(a.queue + 1, 1)] = static_cast<int>(item); };
        const uint32_t z = item / BT, u = item - z * BT;
        const int side = static_cast<int>(z) / a.H, h = static_cast<int>(z) % a.H;
        const int k = a.kk[side];
        const int S = a.S;
        const uint32_t b = u / static_cast<uint32_t>(a.T), t = u - b * static_cast<uint32_t>(a.T);
        const void* X = a.X[side];
        const void* P = a.P[side];
        const int64_t xoff = ((static_cast<int64_t>(b) * a.H + h) * a.T + t) * a.dk;
        const int64_t prow0 = static_cast<int64_t>(h) * 2 * S;

        float e2 = 0.f;
        if (P != nullptr) {
            float ss = 0.f;
            const char* xr = static_cast<const char*>(X) + xoff * D::BYTES;
            if ((reinterpret_cast<uintptr_t>(xr) & 15) == 0 && (a.dk * D::BYTES) % 16 == 0) {
                const int nq = a.dk * D::BYTES / 16;
                for (int q0 = 0; q0 < nq; q0 += 4) {
                    uint4 xq[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (q0 + u < nq) xq[u] = __ldg(reinterpret_cast<const uint4*>(xr) + q0 + u);
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (q0 + u < nq) {
                            float f[D::E];
                            unpack16<D>(xq[u], f);
#pragma unroll
                            for (int e = 0; e < D::E; ++e) ss = fmaf(f[e], f[e], ss);
                        }
                }
            } else {
                for (int d = 0; d < a.dk; ++d) {
                    const float xv = load_elem<D>(X, xoff + d);
                    ss = fmaf(xv, xv, ss);
                }
            }
            e2 = __fmul_ru(__fmul_ru(__fmul_ru(2.f * a.cbound, a.pnorm[side * a.H + h]), sqrtf(ss)), 1.f + 0x1p-12f);
        }

        float amax[2];
        for (int hf = 0; hf < 2; ++hf) {
            const int64_t base = part_at(static_cast<int>(z), 1, hf, BT, u, L, 0);
            float* Av = hf ? A2v : A1v;
            unsigned short* Ai = hf ? A2i : A1i;
            const float4* pv = reinterpret_cast<const float4*>(a.part_v + base);   // L % 4 == 0, 16-byte aligned
            const int4* pi = reinterpret_cast<const int4*>(a.part_i + base);
#pragma unroll
            for (int q4 = 0; q4 < L / 4; ++q4) {
                const float4 v4 = __ldg(pv + q4);
                const int4 i4 = __ldg(pi + q4);
                Av[(4 * q4) * W] = v4.x; Av[(4 * q4 + 1) * W] = v4.y; Av[(4 * q4 + 2) * W] = v4.z; Av[(4 * q4 + 3) * W] = v4.w;
                Ai[(4 * q4) * W] = static_cast<unsigned short>(i4.x); Ai[(4 * q4 + 1) * W] = static_cast<unsigned short>(i4.y);
                Ai[(4 * q4 + 2) * W] = static_cast<unsigned short>(i4.z); Ai[(4 * q4 + 3) * W] = static_cast<unsigned short>(i4.w);
            }
            const float vk = Av[(k - 1) * W], vk1 = Av[k * W];
            if (!(S <= k || __fsub_rd(vk, vk1) > e2)) {
                // band of the half boundary
                ++stat_hb;
                const float lo = __fsub_rd(vk, e2), hi = __fadd_ru(vk1, e2);
                if (S > L && Av[(L - 1) * W] >= lo) { defer(); goto next; }
                int cin = 0, m = 0;
                for (int p = 0; p < L; ++p) {        // (-inf padding never enters a band)
                    const float v = Av[p * W];
                    cin += v > hi ? 1 : 0;
                    m += (v >= lo && v <= hi && v != -INFINITY) ? 1 : 0;
                }
                if (m > BT_BAND) { defer(); goto next; }
                stat_he += m;
                for (int e = 0; e < m; ++e) {
                    const FF f = ff_score_thread<D>(P, X, xoff, prow0, a.dk, S, hf, Ai[(cin + e) * W]);
                    bh[e * W] = f.h; bl[e * W] = f.l; bb[e * W] = f.b;
                }
                bool unsure = false;
                for (int e = 0; e < m; ++e) {
                    const FF fe{bh[e * W], bl[e * W], bb[e * W]};
                    const int ie = Ai[(cin + e) * W];
                    int rank = 0;
                    for (int f = 0; f < m; ++f) {
                        if (f == e) continue;
                        const FF ff{bh[f * W], bl[f * W], bb[f * W]};
                        const int c = ff_cmp(ff, fe, unsure);
                        rank += (c > 0 || (c == 0 && Ai[(cin + f) * W] < ie)) ? 1 : 0;
                    }
                    bc[e * W] = rank < k - cin ? 1 : 0;
                }
                if (unsure) { defer(); goto next; }
                // chosen band entries, in list order, after the certain prefix
                int q2 = cin;
                for (int e = 0; e < m; ++e) {
                    if (bc[e * W]) {
                        const float v = Av[(cin + e) * W];
                        const int ix = Ai[(cin + e) * W];
                        Av[q2 * W] = v; Ai[q2 * W] = static_cast<unsigned short>(ix);   // q2 <= cin + e: in place
                        ++q2;
                    }
                }
            }
            amax[hf] = fmaxf(fabsf(Av[0]), fabsf(Av[(k - 1) * W]));
        }
        {
            const float e2c = __fadd_ru(__fmul_ru(2.f, e2), __fmul_ru(0x1p-21f, __fadd_ru(amax[0], amax[1])));
            // outer-sum candidates by a max-heap of the row heads (k+4 of them, 64 if the band needs)
            const float a20 = A2v[0];
            for (int i = 0; i < k; ++i) { hv[i * W] = A1v[i * W] + a20; hp[i * W] = static_cast<unsigned short>(i); }
            const int kk2 = k * k;
            int npop = 0;
            auto pops = [&](int upto) {
                for (; npop < upto; ++npop) {
                    const float v = hv[0];
                    const int pk = hp[0];
                    const int i = pk & 255, j = pk >> 8;
                    ov[npop * W] = v;
                    os[npop * W] = (j < k) ? A1i[i * W] * S + A2i[j * W] : INT_MAX;
                    const int j1 = j + 1;
                    const float nv = j1 < k ? A1v[i * W] + A2v[j1 * W] : -INFINITY;
                    const int np = i | (j1 << 8);
                    int pos = 0;
                    bool stop = false;
#pragma unroll
                    for (int lvl = 0; lvl < LOG; ++lvl) {
                        const int c = 2 * pos + 1;
                        const float v1 = c < k ? hv[c * W] : -INFINITY;
                        const float v2 = c + 1 < k ? hv[(c + 1) * W] : -INFINITY;
                        const int cm = v2 > v1 ? c + 1 : c;
                        const float vm = fmaxf(v1, v2);
                        if (!stop && vm > nv) { hv[pos * W] = vm; hp[pos * W] = hp[cm * W]; pos = cm; }
                        else stop = true;
                    }
                    hv[pos * W] = nv;
                    hp[pos * W] = static_cast<unsigned short>(np);
                }
            };
            const int len0 = kk2 < L ? kk2 : L;
            pops(len0 > k + 1 ? len0 : k + 1);
            int len = npop;
            const float ck = ov[(k - 1) * W], ck1 = k < npop ? ov[k * W] : -INFINITY;
            int nsel = k;                              // selected: candidates [0, k) unless a band is resolved
            if (!(ck1 == -INFINITY || __fsub_rd(ck, ck1) > e2c)) {
                ++stat_cb;
                const float lo = __fsub_rd(ck, e2c), hi = __fadd_ru(ck1, e2c);
                // a band reaching the last kept candidate (merge to be extended): queue B
                const bool all_cands = len >= kk2;
                if (!all_cands && ov[(len - 1) * W] != -INFINITY && ov[(len - 1) * W] >= lo) { defer(); goto next; }
                int cin = 0, m = 0;
                for (int p = 0; p < len; ++p) {      // (exhausted rows, -inf, never enter a band)
                    const float v = ov[p * W];
                    cin += v > hi ? 1 : 0;
                    m += (v >= lo && v <= hi && v != -INFINITY) ? 1 : 0;
                }
                if (m > BT_BAND) { defer(); goto next; }
                stat_ce += m;
                for (int e = 0; e < m; ++e) {
                    const int f = os[(cin + e) * W];
                    const FF s1 = ff_score_thread<D>(P, X, xoff, prow0, a.dk, S, 0, f / S);
                    const FF s2 = ff_score_thread<D>(P, X, xoff, prow0, a.dk, S, 1, f % S);
                    const FF sm = ff_add(s1, s2, P == nullptr);
                    bh[e * W] = sm.h; bl[e * W] = sm.l; bb[e * W] = sm.b;
                }
                bool unsure = false;
                for (int e = 0; e < m; ++e) {
                    const FF fe{bh[e * W], bl[e * W], bb[e * W]};
                    const int ie = os[(cin + e) * W];
                    int rank = 0;
                    for (int f = 0; f < m; ++f) {
                        if (f == e) continue;
                        const FF ff{bh[f * W], bl[f * W], bb[f * W]};
                        const int c = ff_cmp(ff, fe, unsure);
                        rank += (c > 0 || (c == 0 && os[(cin + f) * W] < ie)) ? 1 : 0;
                    }
                    bc[e * W] = rank < k - cin ? 1 : 0;
                }
                if (unsure) { defer(); goto next; }
                int q2 = cin;
                for (int e = 0; e < m; ++e) {
                    if (bc[e * W]) {
                        const float v = ov[(cin + e) * W];
                        const int f = os[(cin + e) * W];
                        ov[q2 * W] = v; os[q2 * W] = f;
                        ++q2;
                    }
                }
                nsel = q2;                             // = k
            }
            // softmax over the k selected scores, then ascending slot order
            float vmax = -INFINITY;
            for (int r = 0; r < nsel; ++r) vmax = fmaxf(vmax, ov[r * W]);
            float ew[KM];
            int sl[KM];
            float zsum = 0.f;
#pragma unroll
            for (int r = 0; r < KM; ++r) {
                if (r < k) { ew[r] = expf(ov[r * W] - vmax); sl[r] = os[r * W]; zsum += ew[r]; }
                else { ew[r] = 0.f; sl[r] = INT_MAX; }
            }
#pragma unroll
            for (int size = 2; size <= KM; size <<= 1)
#pragma unroll
                for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
                    for (int i = 0; i < KM; ++i) {
                        const int jx = i ^ stride;
                        if (jx > i) {
                            const bool up = (i & size) == 0;
                            const bool sw = up ? (sl[i] > sl[jx]) : (sl[i] < sl[jx]);
                            const int si = sl[i];
                            const float ei = ew[i];
                            sl[i] = sw ? sl[jx] : si;  ew[i] = sw ? ew[jx] : ei;
                            sl[jx] = sw ? si : sl[jx]; ew[jx] = sw ? ei : ew[jx];
                        }
                    }
            const int64_t tokoff = ((static_cast<int64_t>(b) * a.H + h) * a.T + t) * k;
            int32_t* oi = a.idx[side] + tokoff;
            float* ow = a.w[side] + tokoff;
#pragma unroll
            for (int r = 0; r < KM; ++r)
                if (r < k) { oi[r] = sl[r]; ow[r] = ew[r] / zsum; }
        }
    next:;
    }
    if (stat_hb) stat_add(a.err, STAT_HALF_BAND, stat_hb);
    if (stat_he) stat_add(a.err, STAT_HALF_BAND_ENTRIES, stat_he);
    if (stat_cb) stat_add(a.err, STAT_COMB_BAND, stat_cb);
    if (stat_ce) stat_add(a.err, STAT_COMB_BAND_ENTRIES, stat_ce);
}

template <class D, int L>
static cudaError_t launch_finalize(const AddrArgs& a, cudaStream_t stream) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    dim3 gB(static_cast<unsigned>((BT + F_THREADS - 1) / F_THREADS), 2 * a.H);
    cudaError_t e;
    if constexpr (L <= 36) {
        int dev = 0, sms = 0, per_sm = 0;
        e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_addr_finalize<D, L, FIN_FAST>, FW_WARPS * 32, 0);
        if (e != cudaSuccess) return e;
        const int64_t need = (2 * a.H * BT + FW_WARPS - 1) / FW_WARPS;
        const int64_t full = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
        const unsigned grid = static_cast<unsigned>(need < full ? need : full);
        // same carveout as the tensor-core kernel and the M0 copy: they share SMs
        for (auto fn : {k_addr_finalize<D, L, FIN_FAST>, k_addr_finalize<D, L, FIN_BAND>, k_addr_finalize<D, L, FIN_FULL>}) {
            e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
            if (e != cudaSuccess) return e;
        }
        if (a.queue != nullptr) {
            e = cudaMemsetAsync(a.queue, 0, 2 * sizeof(int), stream);
            if (e != cudaSuccess) return e;
            if (a.ncc == 1) {                    // certified pass, one thread per token-side
                const size_t smt = static_cast<size_t>(ft_bytes(L - 4)) * FT_THREADS;
                e = cudaFuncSetAttribute(k_addr_finalize_thread<D, L>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smt));
                if (e != cudaSuccess) return e;
                const int64_t items = 2 * a.H * BT;
                k_addr_finalize_thread<D, L><<<static_cast<unsigned>((items + FT_THREADS - 1) / FT_THREADS), FT_THREADS,
                                               smt, stream>>>(a);
            } else {
                k_addr_finalize<D, L, FIN_FAST><<<grid, FW_WARPS * 32, 0, stream>>>(a);
            }
            // band pass: one thread per queued token-side on large problems; a warp per item when
            // the problem is small (decode): there the queue is short and each item's serial
            // rescoring, not the item count, sets the pass's length
            if (a.ncc == 1 && 2 * a.H * BT >= 32768) {
                const size_t smb = static_cast<size_t>(bt_bytes(L)) * BT_THREADS;
                e = cudaFuncSetAttribute(k_addr_band_thread<D, L>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smb));
                if (e != cudaSuccess) return e;
                const int64_t items = 2 * a.H * BT;       // upper bound of the queue length
                int per_sm_b = 0;
                e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_b, k_addr_band_thread<D, L>, BT_THREADS, smb);
                if (e != cudaSuccess) return e;
                const int64_t need_b = (items + BT_THREADS - 1) / BT_THREADS;
                const int64_t full_b = static_cast<int64_t>(sms) * (per_sm_b > 0 ? per_sm_b : 1);
                k_addr_band_thread<D, L><<<static_cast<unsigned>(need_b < full_b ? need_b : full_b), BT_THREADS,
                                           smb, stream>>>(a);
            } else {
                k_addr_finalize<D, L, FIN_BAND><<<grid, FW_WARPS * 32, 0, stream>>>(a);
            }
        }
        k_addr_finalize<D, L, FIN_FULL><<<grid, FW_WARPS * 32, 0, stream>>>(a);
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
        cudaError_t e = cudaMemsetAsync(a.pnorm, 0, static_cast<size_t>(2) * a.H * sizeof(float), stream);
        if (e != cudaSuccess) return e;
        const int64_t rows = static_cast<int64_t>(2) * a.H * 2 * a.S;
        k_pnorm<D><<<static_cast<unsigned>((rows + 31) / 32), 256, 0, stream>>>(a);
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
