// Hazard pass of the recurrence (K-REC).  The recurrence gathers rows several tokens ahead,
// and several warps advance the tokens of a chain together, so every gather and write is
// checked against the other tokens of a window of LA tokens before it:
//   * read after write: for every (t, n) the latest writer t - delta of the slot, and its
//     position n' in the writer's slot list, for delta in [1, LA] (write-gather) and [0, LA]
//     (read-gather; delta = 0 is a slot the token reads after writing it);
//   * write after read: for every write slot of t, the latest token of [t - LA, t - 1] that
//     read-gathers it.
// This is the sorted-list matching of App. A.2 posed as a lookup: the write and read entries
// of a window of tokens go into a shared-memory hash table keyed by slot, and every access of
// the tile probes it, so the cost does not grow with LA.
#include "sdm_internal.h"

namespace sdm {

// ------------------------------------------------------------------------------------------
// Output: hz[(chain*T + t)*kmax + n], the hazard word of sdm_internal.h (codes, fresh flags of
// the lazy memory when firstw is given, write-after-read distance).  Slot lists must be
// strictly ascending within each token (checked: status bit 1).
//
// One CTA per (chain, tile of `tile` tokens).  The window's lists are staged in shared memory
// (write lists [u][kw], read lists [u][kr], u = token - w0).  A first pass marks every
// entry's 16-bit hash bucket in a `seen` bitmap and the buckets met twice in a `dup` bitmap;
// only entries of `dup` buckets can take part in a hazard (a slot met once in the window has
// none), so only they go into the table and only their accesses probe it -- a few percent at
// random addressing, which keeps most lookups to one bit test.  A table entry is 16 bits,
// 1 + (u << 7 | q) with q the position in the token's write list (q < kw) or kw + the position
// in its read list, 0 marking an empty entry; the slot an entry stands for is read back from
// the staged lists.  Entries go in with a shared-memory compare-and-swap by linear probing; a
// probe walks the cluster of its slot's hash up to the first empty entry and keeps the latest
// qualifying one.  Warps take tokens and lanes take list positions, so no thread divides.
// ------------------------------------------------------------------------------------------
constexpr int HZ_THREADS = 256;
constexpr int HZ_WARPS = HZ_THREADS / 32;
constexpr size_t HZ_SMEM_TARGET = 64 * 1024;       // shared bytes per CTA aimed for
constexpr int HZ_BUCKET_BITS = 16;                  // hash buckets of the seen / dup bitmaps
constexpr int HZ_BITMAP_WORDS = (1 << HZ_BUCKET_BITS) / 32;

__host__ __device__ inline int hz_table_log2(int tile, int la, int kw, int kr) {
    const int entries = (tile + la) * (kw + kr);
    int lg = 6;
    while ((1 << lg) < 2 * entries) ++lg;           // load factor <= 1/2
    return lg;
}

// Shared memory of a CTA: the table (16-bit entries), the seen and dup bitmaps, then the
// window's slot lists as int32.
__host__ __device__ inline size_t hz_smem_bytes(int tile, int la, int kw, int kr) {
    return (static_cast<size_t>(2) << hz_table_log2(tile, la, kw, kr)) + 2 * HZ_BITMAP_WORDS * 4 +
           static_cast<size_t>(tile + la) * (kw + kr) * 4;
}

// Largest tile (64, 32 or 16 tokens) whose shared memory fits the target size.
int hz_tile(int la, int kw, int kr) {
    for (int tile = 64; tile > 16; tile >>= 1)
        if (hz_smem_bytes(tile, la, kw, kr) <= HZ_SMEM_TARGET) return tile;
    return 16;
}

__device__ __forceinline__ uint32_t hz_hash(uint32_t s, int lg) { return (s * 0x9E3779B1u) >> (32 - lg); }
__device__ __forceinline__ uint32_t hz_bucket(uint32_t s) { return ((s ^ (s >> 15)) * 0x85EBCA6Bu) >> (32 - HZ_BUCKET_BITS); }

__global__ void __launch_bounds__(HZ_THREADS, 1) k_hazard(const RecArgs a, int LA, int kmax, int tile, int32_t* hz,
                                                       const int32_t* __restrict__ firstw) {
    extern __shared__ __align__(16) unsigned short tab[];
    const int kw = a.kw, kr = a.kr, kk = kw + kr;
    const int lg = hz_table_log2(tile, LA, kw, kr);
    const uint32_t mask = (1u << lg) - 1u;
    const int ntiles = (a.T + tile - 1) / tile;
    const int64_t chain = blockIdx.x / ntiles;
    const int t0 = static_cast<int>(blockIdx.x - chain * ntiles) * tile;
    const int t1 = min(a.T, t0 + tile);
    const int w0 = max(0, t0 - LA);                         // first token of the window
    const int nu = t1 - w0;                                 // window tokens (<= 94 < 128)
    const int64_t tokbase = chain * a.T;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t* seen = reinterpret_cast<uint32_t*>(tab + (mask + 1));  // [HZ_BITMAP_WORDS]
    uint32_t* dup = seen + HZ_BITMAP_WORDS;                          // [HZ_BITMAP_WORDS]
    int32_t* sw = reinterpret_cast<int32_t*>(dup + HZ_BITMAP_WORDS); // [nu][kw]
    int32_t* sr = sw + nu * kw;                                      // [nu][kr]

    // stage the lists (contiguous per chain: one block of each), clear the table
    {
        const int nw = nu * kw, nr = nu * kr;
        const int32_t* gw = a.idx_w + (tokbase + w0) * kw;
        const int32_t* gr = a.idx_r + (tokbase + w0) * kr;
        const bool v4 = ((reinterpret_cast<uintptr_t>(gw) | reinterpret_cast<uintptr_t>(gr)) & 15) == 0 && nw % 4 == 0 && nr % 4 == 0;
        if (v4) {
            for (int i = threadIdx.x; i < nw / 4; i += HZ_THREADS) reinterpret_cast<int4*>(sw)[i] = __ldg(reinterpret_cast<const int4*>(gw) + i);
            for (int i = threadIdx.x; i < nr / 4; i += HZ_THREADS) reinterpret_cast<int4*>(sr)[i] = __ldg(reinterpret_cast<const int4*>(gr) + i);
        } else {
            for (int i = threadIdx.x; i < nw; i += HZ_THREADS) sw[i] = __ldg(gw + i);
            for (int i = threadIdx.x; i < nr; i += HZ_THREADS) sr[i] = __ldg(gr + i);
        }
        // table and both bitmaps are contiguous: (mask + 1) * 2 + 2 * HZ_BITMAP_WORDS * 4 bytes
        const int nclr = static_cast<int>(((mask + 1) * 2 + 2 * HZ_BITMAP_WORDS * 4) / 16);
        for (int i = threadIdx.x; i < nclr; i += HZ_THREADS) reinterpret_cast<uint4*>(tab)[i] = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    // mark the buckets of the window's entries: seen once, then dup
    for (int uo = warp; uo < nu; uo += HZ_WARPS) {
        for (int q = lane; q < kk; q += 32) {
            const uint32_t hb = hz_bucket(static_cast<uint32_t>(q < kw ? sw[uo * kw + q] : sr[uo * kr + (q - kw)]));
            const uint32_t bit = 1u << (hb & 31);
            if (atomicOr(seen + (hb >> 5), bit) & bit) atomicOr(dup + (hb >> 5), bit);
        }
    }
    __syncthreads();
    // insert the entries of dup buckets of tokens [w0, t1): warp per token, lane per position
    for (int uo = warp; uo < nu; uo += HZ_WARPS) {
        for (int q = lane; q < kk; q += 32) {
            const int32_t s = q < kw ? sw[uo * kw + q] : sr[uo * kr + (q - kw)];
            const uint32_t hb = hz_bucket(static_cast<uint32_t>(s));
            if (!(dup[hb >> 5] & (1u << (hb & 31)))) continue;
            const unsigned short en = static_cast<unsigned short>(1 + ((uo << 7) | q));
            uint32_t h = hz_hash(static_cast<uint32_t>(s), lg);
            for (uint32_t probe = 0; probe <= mask; ++probe) {      // the table is never full
                if (atomicCAS(tab + h, static_cast<unsigned short>(0), en) == 0) break;
                h = (h + 1) & mask;
            }
        }
    }
    __syncthreads();
    // probe for every access of the tile's tokens: warp per token, lane per position
    const uint32_t N = static_cast<uint32_t>(a.N);
    bool unsorted = false;
    for (int t = t0 + warp; t < t1; t += HZ_WARPS) {
        const int64_t tok = tokbase + t;
        for (int n = lane; n < kmax; n += 32) {
            int word_out = 0;
#pragma unroll
            for (int side = 0; side < 2; ++side) {                  // 0: write slot, 1: read slot
                const int k = side ? kr : kw;
                if (n >= k) continue;
                const int32_t* lst = (side ? sr + (t - w0) * kr : sw + (t - w0) * kw);
                const int32_t s = lst[n];
                if (n > 0 && lst[n - 1] >= s) unsorted = true;
                const int hi = side ? t : t - 1;                     // writers u in [t - LA, hi]
                int best_w = -1, best_n = 0, best_r = -1;
                const uint32_t hb = hz_bucket(static_cast<uint32_t>(s));
                const bool maybe = (dup[hb >> 5] >> (hb & 31)) & 1u;
                uint32_t h = hz_hash(static_cast<uint32_t>(s), lg);
                for (uint32_t probe = 0; maybe && probe <= mask; ++probe) {
                    const int en = tab[h];
                    if (en == 0) break;
                    const int uo = (en - 1) >> 7, q = (en - 1) & 127;
                    const bool rd = q >= kw;
                    const int32_t sv = rd ? sr[uo * kr + (q - kw)] : sw[uo * kw + q];
                    if (sv == s) {
                        const int u = w0 + uo;
                        if (rd) {
                            if (side == 0 && u >= t - LA && u <= t - 1 && u > best_r) best_r = u;
                        } else if (u >= t - LA && u <= hi && u > best_w) {
                            best_w = u;
                            best_n = q;
                        }
                    }
                    h = (h + 1) & mask;
                }
                int c = best_w >= 0 ? 1 + (t - best_w) * 64 + best_n : 0;
                if (firstw && static_cast<uint32_t>(s) < N && __ldg(firstw + chain * a.N + s) >= t)
                    c |= side ? (HZ_R_FRESH >> HZ_R_SHIFT) : HZ_W_FRESH;
                word_out |= side ? c << HZ_R_SHIFT : c;
                if (side == 0 && best_r >= 0) word_out |= (t - best_r) << HZ_WAR_SHIFT;
            }
            hz[tok * kmax + n] = word_out;
        }
    }
    if (__syncthreads_or(unsorted) && threadIdx.x == 0) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_hazard(const RecArgs& a, int la, int kmax, int32_t* hz, cudaStream_t stream, const int32_t* firstw) {
    if (la > HZ_MAX_LA || a.kw + a.kr > 128) return cudaErrorInvalidValue;
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    const int tile = hz_tile(la, a.kw, a.kr);
    const int ntiles = (a.T + tile - 1) / tile;
    const size_t smem = hz_smem_bytes(tile, la, a.kw, a.kr);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_hazard, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    k_hazard<<<static_cast<unsigned>(chains * ntiles), HZ_THREADS, smem, stream>>>(a, la, kmax, tile, hz, firstw);
    return cudaGetLastError();
}

}  // namespace sdm
