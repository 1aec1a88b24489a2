// Hazard pass of the recurrence (K-REC).  The recurrence prefetches the rows token t will
// gather LA tokens ahead; a prefetched row is stale when a token in between wrote that
// slot.  For every (t, n) this pass finds the most recent writer t - delta of the slot and
// its position n' in the writer's (ascending) slot list -- the sorted-list matching of
// App. A.2, done as a binary search -- for delta in [1, LA] (write-gather) and [0, LA]
// (read-gather; delta = 0 is a slot the token reads after writing it).
#include "sdm_internal.h"

namespace sdm {

// ------------------------------------------------------------------------------------------
// Hazard pass.  hz[(chain*T + t)*kmax + n] = write code (low 16 bits) | read code << 16;
// code 0 = no hazard, else 1 + delta*64 + n' (writer t - delta, position n' of its list),
// delta in [1, LA] for the write-gather and [0, LA] for the read-gather.  Codes stay below
// 2^15; bit 15 of each half marks a fresh slot (lazy initial memory: no token wrote it
// before t, so the gather reads M0's row), set only when firstw is given.
// Slot lists must be ascending within each token (as the addressing produces them).
// ------------------------------------------------------------------------------------------
// One warp per token: lane n holds slot n (and n + 32) of the token's lists; the write list
// of each earlier token in the window is spread one entry per lane and searched with a
// branch-free binary search over lanes (every lane runs the same shuffles), most recent
// token first.  k_write, k_read <= 64.
__device__ __forceinline__ int warp_find(int lo_val, int hi_val, int k, int s) {
    // lower bound of s in the ascending list (entry p in lane p & 31: lo_val if p < 32, else hi_val)
    int pos = 0;
#pragma unroll
    for (int step = 32; step >= 1; step >>= 1) {
        const int idx = pos + step - 1;
        const int vlo = __shfl_sync(0xffffffffu, lo_val, idx & 31);
        const int vhi = __shfl_sync(0xffffffffu, hi_val, idx & 31);
        const int v = idx < 32 ? vlo : vhi;
        if (idx < k && v < s) pos += step;
    }
    const int vlo = __shfl_sync(0xffffffffu, lo_val, pos & 31);
    const int vhi = __shfl_sync(0xffffffffu, hi_val, pos & 31);
    const int v = pos < 32 ? vlo : vhi;
    return (pos < k && v == s) ? pos : -1;
}

__global__ void __launch_bounds__(256) k_hazard(const RecArgs a, int LA, int kmax, int32_t* hz,
                                                const int32_t* __restrict__ firstw) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.H * a.T;
    const int64_t tok = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (tok >= BT) return;                     // whole warps exit together
    const int64_t chain = tok / a.T;
    const int t = static_cast<int>(tok - chain * a.T);
    const int kw = a.kw, kr = a.kr;
    const int nq = kmax > 32 ? 2 : 1;          // warp-uniform
    const int32_t* iw = a.idx_w + tok * kw;
    const int32_t* ir = a.idx_r + tok * kr;
    int sw[2] = {-1, -1}, sr[2] = {-1, -1};
    bool unsorted = false;
    for (int q = 0; q < nq; ++q) {
        const int n = lane + 32 * q;
        if (n < kw) { sw[q] = __ldg(iw + n); if (n > 0 && __ldg(iw + n - 1) >= sw[q]) unsorted = true; }
        if (n < kr) { sr[q] = __ldg(ir + n); if (n > 0 && __ldg(ir + n - 1) >= sr[q]) unsorted = true; }
    }
    if (__any_sync(0xffffffffu, unsorted) && lane == 0) flag_error(a.err, ERR_UNSORTED);
    int cw[2] = {0, 0}, cr[2] = {0, 0};
    const int dmax = LA < t ? LA : t;          // warp-uniform
    for (int d = 0; d <= dmax; ++d) {
        const int32_t* pw = a.idx_w + (tok - d) * kw;        // write list of token t - d
        const int lo_val = lane < kw ? __ldg(pw + lane) : INT_MAX;
        const int hi_val = lane + 32 < kw ? __ldg(pw + lane + 32) : INT_MAX;
        for (int q = 0; q < nq; ++q) {
            const int pw_pos = warp_find(lo_val, hi_val, kw, sw[q]);
            const int pr_pos = warp_find(lo_val, hi_val, kw, sr[q]);
            if (d >= 1 && cw[q] == 0 && sw[q] >= 0 && pw_pos >= 0) cw[q] = 1 + d * 64 + pw_pos;
            if (cr[q] == 0 && sr[q] >= 0 && pr_pos >= 0) cr[q] = 1 + d * 64 + pr_pos;
        }
    }
    if (firstw) {
        const int32_t* fw = firstw + chain * a.N;
        const uint32_t N = static_cast<uint32_t>(a.N);
        for (int q = 0; q < nq; ++q) {
            if (static_cast<uint32_t>(sw[q]) < N && __ldg(fw + sw[q]) >= t) cw[q] |= 0x8000;
            if (static_cast<uint32_t>(sr[q]) < N && __ldg(fw + sr[q]) >= t) cr[q] |= 0x8000;
        }
    }
    for (int q = 0; q < nq; ++q) {
        const int n = lane + 32 * q;
        if (n < kmax) hz[tok * kmax + n] = cw[q] | (cr[q] << 16);
    }
}

cudaError_t launch_hazard(const RecArgs& a, int la, int kmax, int32_t* hz, cudaStream_t stream, const int32_t* firstw) {
    const int64_t BT = static_cast<int64_t>(a.B) * a.H * a.T;
    k_hazard<<<static_cast<unsigned>((BT + 7) / 8), 256, 0, stream>>>(a, la, kmax, hz, firstw);
    return cudaGetLastError();
}

}  // namespace sdm
