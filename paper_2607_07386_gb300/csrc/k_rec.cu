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
    // widest d-range per warp (<= 128 B) that still gives a few hundred warps
    int dch = 1;
    while (dch < 8 && nch % (dch * 2) == 0) dch *= 2;
    while (dch > 2 && chains * (nch / dch) < 1024) dch /= 2;     // many warps; keep >= 32-byte pieces
    int spt = (kmax + (32 / dch) - 1) / (32 / dch);
    while (spt > 8 && dch > 1) { dch /= 2; spt = (kmax + (32 / dch) - 1) / (32 / dch); }   // k = 64 with wide ranges
    p.dch = dch;
    p.nsplit = nch / dch;
    p.spt = spt <= 1 ? 1 : spt <= 2 ? 2 : spt <= 4 ? 4 : 8;
    p.threads = 32;
    p.la = T <= 1 ? 1 : 4;
    // writer/reader warp pairs: measured faster only with short slot lists (k <= 16) and
    // few units (256 at B=4 H=8 k=16: 1.34 -> 1.12 ms); with k = 32 the hand-over costs more
    // than it saves (1024 units: 4.33 -> 5.69 ms; 256 units, T = 65536: 51.8 -> 55.2 ms)
    p.split = p.la > 1 && kmax <= 16 && chains * p.nsplit < 768;
    p.smem = rec_smem_bytes(p.la, (32 / dch) * p.spt, dch);
    // four consecutive d-ranges of a chain per CTA: an SM then serves the rows of fewer chains,
    // whose gathers hit fewer memory pages (layer_1p4b: 9.83 -> 9.67 ms per broadcast step,
    // 9.41 -> 8.71 ms per lazy step, where the gathers span both mem and M0; 8 per CTA: 9.94
    // and 8.98 ms)
    // (only with enough warps to fill the SMs: long_ctx's 256 warps run 1% slower in 64 CTAs)
    p.wpc = p.la > 1 && p.nsplit % 4 == 0 && chains * p.nsplit >= 512 ? 4 : 1;
    return p;
}

size_t rec_workspace_bytes(int B, int H, int T, int kw, int kr) {
    const int kmax = kw > kr ? kw : kr;
    return static_cast<size_t>(B) * H * T * kmax * sizeof(int32_t);
}

cudaError_t launch_recur(int dtype, const RecArgs& a, int32_t* hz_ws, cudaStream_t stream, const int32_t* firstw) {
    const RecPlan p = rec_plan(dtype, a.B, a.H, a.T, a.dv, a.kw, a.kr);
    cudaError_t e = launch_hazard(a, p.la, p.kmax, hz_ws, stream, a.M0 ? firstw : nullptr);
    if (e != cudaSuccess) return e;
    auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
    const int vec_lists = (a.kw % 4 == 0) && (a.kr % 4 == 0) && (p.kmax % 4 == 0) && al16(a.idx_w) && al16(a.w_w) &&
                          al16(a.idx_r) && al16(a.w_r) && al16(hz_ws);
    return dtype == 0 ? launch_recur_f32(p, a, hz_ws, vec_lists, stream) : launch_recur_bf16(p, a, hz_ws, vec_lists, stream);
}

}  // namespace sdm
