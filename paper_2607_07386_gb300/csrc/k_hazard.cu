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
// One CTA per (chain, tile of `tile` tokens).  Table entries are 64-bit words
//   slot (high 32 bits) | read flag (bit 31) | window token (bits 16-30) | list position (bits 0-15),
// inserted with a shared-memory compare-and-swap by linear probing; a probe walks the cluster
// of its slot's hash up to the first empty word and keeps the latest qualifying entry.
// ------------------------------------------------------------------------------------------
constexpr int HZ_THREADS = 256;
constexpr unsigned long long HZ_EMPTY = ~0ull;
constexpr size_t HZ_TABLE_TARGET = 64 * 1024;      // bytes of table per CTA aimed for

__host__ __device__ inline int hz_table_log2(int tile, int la, int kw, int kr) {
    const int entries = (tile + la) * (kw + kr);
    int lg = 6;
    while ((1 << lg) < 2 * entries) ++lg;
    return lg;
}

// Shared memory of a CTA: the table, then the window's slot lists (write, then read) as int32.
__host__ __device__ inline size_t hz_smem_bytes(int tile, int la, int kw, int kr) {
    return (static_cast<size_t>(8) << hz_table_log2(tile, la, kw, kr)) + static_cast<size_t>(tile + la) * (kw + kr) * 4;
}

// Largest tile (64, 32 or 16 tokens) whose table fits the target size.
int hz_tile(int la, int kw, int kr) {
    for (int tile = 64; tile > 16; tile >>= 1)
        if (hz_smem_bytes(tile, la, kw, kr) <= HZ_TABLE_TARGET + 32 * 1024) return tile;
    return 16;
}


__device__ __forceinline__ uint32_t hz_hash(uint32_t s, int lg) { return (s * 0x9E3779B1u) >> (32 - lg); }

__global__ void __launch_bounds__(HZ_THREADS) k_hazard(const RecArgs a, int LA, int kmax, int tile, int32_t* hz,
                                                       const int32_t* __restrict__ firstw) {
    extern __shared__ unsigned long long tab[];
    const int kw = a.kw, kr = a.kr;
    const int lg = hz_table_log2(tile, LA, kw, kr);
    const uint32_t mask = (1u << lg) - 1u;
    const int ntiles = (a.T + tile - 1) / tile;
    const int64_t chain = blockIdx.x / ntiles;
    const int t0 = static_cast<int>(blockIdx.x - chain * ntiles) * tile;
    const int t1 = min(a.T, t0 + tile);
    const int w0 = max(0, t0 - LA);                         // first token of the window
    const int64_t tokbase = chain * a.T;
    // the window's lists in shared memory: sw [t1 - w0][kw], then sr [t1 - w0][kr]
    int32_t* sw = reinterpret_cast<int32_t*>(tab + (mask + 1));
    int32_t* sr = sw + (t1 - w0) * kw;

    // stage the lists (contiguous per chain: one block of each), clear the table
    {
        const int nw = (t1 - w0) * kw, nr = (t1 - w0) * kr;
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
    }
    for (int i = threadIdx.x; i <= static_cast<int>(mask); i += HZ_THREADS) tab[i] = HZ_EMPTY;
    __syncthreads();
    // insert the write and read entries of tokens [w0, t1)
    const int kk = kw + kr;
    const int nins = (t1 - w0) * kk;
    for (int e = threadIdx.x; e < nins; e += HZ_THREADS) {
        const int u = w0 + e / kk, q = e - (e / kk) * kk;
        const bool rd = q >= kw;
        const int n = rd ? q - kw : q;
        const int32_t s = rd ? sr[(u - w0) * kr + n] : sw[(u - w0) * kw + n];
        const unsigned long long word = (static_cast<unsigned long long>(static_cast<uint32_t>(s)) << 32) |
                                        (rd ? 0x80000000ull : 0ull) |
                                        (static_cast<unsigned long long>(u - w0) << 16) | static_cast<unsigned>(n);
        uint32_t h = hz_hash(static_cast<uint32_t>(s), lg);
        for (uint32_t probe = 0; probe <= mask; ++probe) {          // the table is never full
            if (atomicCAS(&tab[h], HZ_EMPTY, word) == HZ_EMPTY) break;
            h = (h + 1) & mask;
        }
    }
    __syncthreads();
    // probe for every access of the tile's tokens; one thread per (token, position)
    const uint32_t N = static_cast<uint32_t>(a.N);
    bool unsorted = false;
    const int nacc = (t1 - t0) * kmax;
    for (int e = threadIdx.x; e < nacc; e += HZ_THREADS) {
        const int t = t0 + e / kmax, n = e - (e / kmax) * kmax;
        const int64_t tok = tokbase + t;
        int word_out = 0;
#pragma unroll
        for (int side = 0; side < 2; ++side) {                      // 0: write slot, 1: read slot
            const int k = side ? kr : kw;
            if (n >= k) continue;
            const int32_t* lst = (side ? sr : sw) + (t - w0) * k;
            const int32_t s = lst[n];
            if (n > 0 && lst[n - 1] >= s) unsorted = true;
            const int hi = side ? t : t - 1;                         // writers u in [t - LA, hi]
            int best_w = -1, best_n = 0, best_r = -1;
            uint32_t h = hz_hash(static_cast<uint32_t>(s), lg);
            for (uint32_t probe = 0; probe <= mask; ++probe) {
                const unsigned long long word = tab[h];
                if (word == HZ_EMPTY) break;
                if (static_cast<int32_t>(word >> 32) == s) {
                    const int u = w0 + static_cast<int>((word >> 16) & 0x7fff);
                    if (word & 0x80000000ull) {
                        if (side == 0 && u >= t - LA && u <= t - 1 && u > best_r) best_r = u;
                    } else if (u >= t - LA && u <= hi && u > best_w) {
                        best_w = u;
                        best_n = static_cast<int>(word & 0xffff);
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
    if (__syncthreads_or(unsorted) && threadIdx.x == 0) flag_error(a.err, ERR_UNSORTED);
}

cudaError_t launch_hazard(const RecArgs& a, int la, int kmax, int32_t* hz, cudaStream_t stream, const int32_t* firstw) {
    if (la > HZ_MAX_LA) return cudaErrorInvalidValue;
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
