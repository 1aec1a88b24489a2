// Hazard pass of the recurrence (K-REC).  The recurrence prefetches the rows a token will
// gather several tokens ahead; a prefetched row is stale when a token in between wrote that
// slot.  For every (t, n) this pass finds the most recent writer t - delta of the slot and
// its position n' in the writer's slot list, for delta in [1, LA] (write-gather) and [0, LA]
// (read-gather; delta = 0 is a slot the token reads after writing it).  This is the
// sorted-list matching of App. A.2 posed as a lookup: the write entries of a window of
// tokens go into a shared-memory hash table keyed by slot, and every access of the tile
// probes it, so the cost does not grow with the look-ahead LA.
#include "sdm_internal.h"

namespace sdm {

// ------------------------------------------------------------------------------------------
// hz[(chain*T + t)*kmax + n] = write code (low 16 bits) | read code << 16; code 0 = no hazard,
// else 1 + delta*64 + n' (writer t - delta, position n' of its list), delta in [1, LA] for the
// write-gather and [0, LA] for the read-gather.  Codes stay below 2^15 (LA <= 64); bit 15 of
// each half marks a fresh slot (lazy initial memory: no token wrote it before t, so the
// gather reads M0's row), set only when firstw is given.  Slot lists must be strictly
// ascending within each token (checked: status bit 1).
//
// One CTA per (chain, tile of HZ_TILE tokens).  Table entries are 64-bit words
// slot (high 32 bits) | window token (16 bits) | list position (16 bits), inserted with a
// shared-memory compare-and-swap by linear probing; a probe walks the cluster of its
// slot's hash up to the first empty word and keeps the latest qualifying writer.
// ------------------------------------------------------------------------------------------
constexpr int HZ_TILE = 64;
constexpr int HZ_THREADS = 256;
constexpr unsigned long long HZ_EMPTY = ~0ull;

__host__ __device__ inline int hz_table_log2(int la, int kw) {
    const int entries = (HZ_TILE + la) * kw;
    int lg = 6;
    while ((1 << lg) < 2 * entries) ++lg;
    return lg;
}

__device__ __forceinline__ uint32_t hz_hash(uint32_t s, int lg) { return (s * 0x9E3779B1u) >> (32 - lg); }

__global__ void __launch_bounds__(HZ_THREADS) k_hazard(const RecArgs a, int LA, int kmax, int32_t* hz,
                                                       const int32_t* __restrict__ firstw) {
    extern __shared__ unsigned long long tab[];
    const int lg = hz_table_log2(LA, a.kw);
    const uint32_t mask = (1u << lg) - 1u;
    const int ntiles = (a.T + HZ_TILE - 1) / HZ_TILE;
    const int64_t chain = blockIdx.x / ntiles;
    const int t0 = static_cast<int>(blockIdx.x - chain * ntiles) * HZ_TILE;
    const int t1 = min(a.T, t0 + HZ_TILE);
    const int w0 = max(0, t0 - LA);                         // first token of the window
    const int kw = a.kw, kr = a.kr;
    const int64_t tokbase = chain * a.T;

    for (int i = threadIdx.x; i <= static_cast<int>(mask); i += HZ_THREADS) tab[i] = HZ_EMPTY;
    __syncthreads();
    // insert the write entries of tokens [w0, t1)
    const int nins = (t1 - w0) * kw;
    for (int e = threadIdx.x; e < nins; e += HZ_THREADS) {
        const int u = w0 + e / kw, n = e - (e / kw) * kw;
        const int32_t s = __ldg(a.idx_w + (tokbase + u) * kw + n);
        const unsigned long long word = (static_cast<unsigned long long>(static_cast<uint32_t>(s)) << 32) |
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
        int code[2] = {0, 0};
#pragma unroll
        for (int side = 0; side < 2; ++side) {                      // 0: write-gather, 1: read-gather
            const int k = side ? kr : kw;
            if (n >= k) continue;
            const int32_t* lst = (side ? a.idx_r : a.idx_w) + tok * k;
            const int32_t s = __ldg(lst + n);
            if (n > 0 && __ldg(lst + n - 1) >= s) unsorted = true;
            const int lo = t - LA, hi = side ? t : t - 1;            // writers u in [lo, hi]
            int best_u = -1, best_n = 0;
            uint32_t h = hz_hash(static_cast<uint32_t>(s), lg);
            for (uint32_t probe = 0; probe <= mask; ++probe) {
                const unsigned long long word = tab[h];
                if (word == HZ_EMPTY) break;
                if (static_cast<int32_t>(word >> 32) == s) {
                    const int u = w0 + static_cast<int>((word >> 16) & 0xffff);
                    if (u >= lo && u <= hi && u > best_u) { best_u = u; best_n = static_cast<int>(word & 0xffff); }
                }
                h = (h + 1) & mask;
            }
            int c = best_u >= 0 ? 1 + (t - best_u) * 64 + best_n : 0;
            if (firstw && static_cast<uint32_t>(s) < N && __ldg(firstw + chain * a.N + s) >= t) c |= 0x8000;
            code[side] = c;
        }
        hz[tok * kmax + n] = code[0] | (code[1] << 16);
    }
    if (__syncthreads_or(unsorted) && threadIdx.x == 0) flag_error(a.err, ERR_UNSORTED);
}

size_t hazard_smem_bytes(int la, int kw) { return (static_cast<size_t>(1) << hz_table_log2(la, kw)) * 8; }

cudaError_t launch_hazard(const RecArgs& a, int la, int kmax, int32_t* hz, cudaStream_t stream, const int32_t* firstw) {
    const int64_t chains = static_cast<int64_t>(a.B) * a.H;
    const int ntiles = (a.T + HZ_TILE - 1) / HZ_TILE;
    const size_t smem = hazard_smem_bytes(la, a.kw);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_hazard, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    k_hazard<<<static_cast<unsigned>(chains * ntiles), HZ_THREADS, smem, stream>>>(a, la, kmax, hz, firstw);
    return cudaGetLastError();
}

}  // namespace sdm
