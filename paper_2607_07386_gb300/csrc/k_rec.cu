// K-REC host side: launch geometry, scratch size, hazard pass + recurrence launch.
// Kernels: k_rec_impl.cuh (recurrence, instantiated in k_rec_bf16.cu / k_rec_f32.cu) and
// k_hazard.cu (hazard pass).
#include "k_rec_impl.cuh"

namespace sdm {

cudaError_t launch_recur_bf16(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s);
cudaError_t launch_recur_f32(const RecPlan& p, const RecArgs& a, const int32_t* hz, int vec_lists, cudaStream_t s);
cudaError_t launch_hazard(const RecArgs& a, int la, int kmax, int32_t* hz, cudaStream_t stream, const int32_t* firstw);

RecPlan rec_plan(int dtype, int B, int H, int T, int dv, int kw, int kr) {
    RecPlan p{};
    const int bytes = dtype == 0 ? 4 : 2;
    const int nch = dv * bytes / 16;                       // 16-byte chunks per row
    const int64_t chains = static_cast<int64_t>(B) * H;
    const int kmax = kw > kr ? kw : kr;
    p.kmax = kmax;
    if (T <= 1) {
        // one token per chain: one warp per (chain, d-range), widest d-range (<= 128 B) that
        // still gives a thousand warps; no look-ahead
        int dch = 1;
        while (dch < 8 && nch % (dch * 2) == 0) dch *= 2;
        while (dch > 2 && chains * (nch / dch) < 1024) dch /= 2;
        int spt = (kmax + (32 / dch) - 1) / (32 / dch);
        while (spt > 8 && dch > 1) { dch /= 2; spt = (kmax + (32 / dch) - 1) / (32 / dch); }
        p.dch = dch;
        p.nsplit = nch / dch;
        p.spt = spt <= 1 ? 1 : spt <= 2 ? 2 : spt <= 4 ? 4 : 8;
        p.la = 1;
        p.w = 0;
        p.p = 1;
        return p;
    }
    // token-interleaved kernel: W warps per (chain, d-range) CTA, each prefetching P = 2 of
    // its own tokens ahead.  64-byte d-ranges (four lanes per slot row) keep the per-token
    // work of each warp small; W = 8 and 32-byte d-ranges when the chains alone give fewer
    // than 2048 warps (long sequences on few chains).
    int dch = 1;
    while (dch < 4 && nch % (dch * 2) == 0) dch *= 2;
    int w = 4;
    if (chains * (nch / dch) * w < 2048) w = 8;
    while (dch > 2 && chains * (nch / dch) * w < 2048) dch /= 2;
    int spt = (kmax + (32 / dch) - 1) / (32 / dch);
    while (spt > 8 && dch > 1) { dch /= 2; spt = (kmax + (32 / dch) - 1) / (32 / dch); }
    p.dch = dch;
    p.nsplit = nch / dch;
    p.spt = spt <= 1 ? 1 : spt <= 2 ? 2 : spt <= 4 ? 4 : 8;
    p.w = w;
    p.p = 2;
    p.la = (p.p + 1) * w;
    return p;
}

size_t rec_workspace_bytes(int B, int H, int T, int kw, int kr) {
    const int kmax = kw > kr ? kw : kr;
    return static_cast<size_t>(B) * H * T * kmax * sizeof(int32_t);
}

cudaError_t launch_recur(int dtype, const RecArgs& a_in, int32_t* hz_ws, cudaStream_t stream, const int32_t* firstw,
                         cudaEvent_t mem_ready) {
    RecArgs a = a_in;
    a.firstw = a.M0 ? firstw : nullptr;
    const RecPlan p = rec_plan(dtype, a.B, a.H, a.T, a.dv, a.kw, a.kr);
    if (p.w > 0) {                 // one token per chain needs no hazard table
        cudaError_t e = launch_hazard(a, p.la, p.kmax, hz_ws, stream, a.firstw);
        if (e != cudaSuccess) return e;
    }
    if (mem_ready != nullptr) {    // the hazard pass reads no memory rows: only the recurrence waits
        cudaError_t e = cudaStreamWaitEvent(stream, mem_ready, 0);
        if (e != cudaSuccess) return e;
    }
    auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
    const int vec_lists = (a.kw % 4 == 0) && (a.kr % 4 == 0) && (p.kmax % 4 == 0) && al16(a.idx_w) && al16(a.w_w) &&
                          al16(a.idx_r) && al16(a.w_r) && al16(hz_ws);
    return dtype == 0 ? launch_recur_f32(p, a, hz_ws, vec_lists, stream) : launch_recur_bf16(p, a, hz_ws, vec_lists, stream);
}

}  // namespace sdm
