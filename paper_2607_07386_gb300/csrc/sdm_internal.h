// Host-side interface between the C ABI (sdm_api.cu) and the kernel translation units.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>
#include <stddef.h>

#include "sdm.h"
#include "sdm_common.cuh"

namespace sdm {

// ---------------------------------------------------------------- K-INIT
// ctas_per_sm: 8 fills the SMs (the copy alone); fewer leave room for kernels running beside it.
cudaError_t launch_init_memory(const void* M0, void* mem, int64_t bytes_per_seq, int B, cudaStream_t stream,
                               int ctas_per_sm = 8);
// The same broadcast through the bulk-copy engine (one thread per SM; bytes_per_seq a multiple
// of 16, both pointers 16-byte aligned); a bounded wait that runs out sets ERR_TIMEOUT.
cudaError_t launch_init_bulk(const void* M0, void* mem, int64_t bytes_per_seq, int B, int* err, cudaStream_t stream);

// ---------------------------------------------------------------- K-ADDR
// "which" 0 = read side (q with P_q -> idx_r, w_r), 1 = write side (k with P_k -> idx_w, w_w).
struct AddrArgs {
    const void* P[2];      // [H, 2S, dk] per side, or nullptr (DIRECT mode: scores are x)
    const void* X[2];      // [B, H, T, dk]
    int32_t* idx[2];       // [B, H, T, k_side]
    float* w[2];           // [B, H, T, k_side]
    int kk[2];             // k_read, k_write
    int B, H, T, dk, S;
    int ncc;               // column chunks per half
    int cw;                // columns per chunk (the last one may be shorter)
    float cbound;          // |fp32 score - float64 score| <= cbound * max_j ||P_j|| * ||x||
    float* part_v;         // workspace [2H][2 ncc][L][B*T]: per-chunk top-L scores
    int* part_i;           //   ... and their column index within the half
    float* pnorm;          // workspace [2H]: max row norm of P per side and head
    int* queue;            // workspace [2 + 2 (2 H B T)]: counts of queues A and B, then their
                           // token-side ids (nullptr: one pass does everything)
    int* err;              // device status word
    float* raw;            // test hook of the tensor-core score kernel: raw fp32 scores
                           // [2H][B*T][2S] instead of the per-chunk lists (nullptr normally)
};

// Geometry of the PKM partial lists for a shape (depends only on the shape).
struct AddrPlan {
    int L;      // list length kept per chunk (>= k + 4)
    int ncc;    // column chunks per half
    int cw;     // columns per chunk (<= 512)
    bool mma;   // scores on the tensor cores (bf16, PROJECTED, d_k <= 128, k <= 32)
};
AddrPlan addr_plan(int dtype, int direct, int B, int H, int T, int dk, int S, int kmax);
bool mma_path_supported(int dtype, int direct, int dk, int S, int kmax);
cudaError_t launch_address_mma(const AddrPlan& plan, const AddrArgs& a, cudaStream_t stream);
size_t addr_partial_bytes(const AddrPlan& plan, int B, int H, int T);
size_t addr_queue_bytes(int B, int H, int T);
cudaError_t launch_address(int dtype, const AddrPlan& plan, const AddrArgs& a, cudaStream_t stream);

// ---------------------------------------------------------------- K-REC
struct RecArgs {
    const int32_t* idx_w; const float* w_w;   // [B, H, T, kw]
    const int32_t* idx_r; const float* w_r;   // [B, H, T, kr]
    const void* v;                            // [B, H, T, dv]
    const void* alpha; const void* beta;      // [B, H, T]
    void* mem;                                // [B, H, N, dv]
    const void* M0;                           // [H, N, dv]: source of fresh rows (lazy initial
                                              // memory), or nullptr
    void* undo;                               // [B, H, T, kw, dv]: rows each write overwrote (the
                                              // backward's undo log), or nullptr
    void* y;                                  // [B, H, T, dv]
    int B, H, T, dv, kw, kr;
    int64_t N;
    int* err;
    const int32_t* firstw;                    // lazy initial memory: first writer of each slot in
                                              // this call ([B*H, N]), or nullptr
    long long wait_cycles;                    // limit of every bounded device wait (0: the default)
    int hold_handover;                        // test hook: the first warp withholds its first
                                              // progress word, so the other warps' waits run out
};
// Hazard word of a (token t, list position n) pair: written by the hazard pass (k_hazard.cu),
// read by the recurrence kernels.
//   bits  0-10  write-gather code: 0 = no token of the window [t - LA, t - 1] wrote the slot,
//               else 1 + delta * 64 + n' (the latest writer t - delta, its list position n')
//   bit   11    the write slot is fresh (lazy memory: not written before t; gather M0's row)
//   bits 12-22  read-gather code, as above with delta in [0, LA] (delta = 0: this token)
//   bit   23    the read slot is fresh
//   bits 24-29  write after read: t - u for the latest token u of the window that
//               read-gathers the write slot (0: none)
constexpr int HZ_CODE_MASK = 0x7ff;
constexpr int HZ_W_FRESH = 1 << 11;
constexpr int HZ_R_SHIFT = 12;
constexpr int HZ_R_FRESH = 1 << 23;
constexpr int HZ_WAR_SHIFT = 24;
constexpr int HZ_MAX_LA = 30;           // 1 + 30 * 64 + 63 < 2^11, and distances < 64
__host__ __device__ __forceinline__ int hz_wcode(int h) { return h & HZ_CODE_MASK; }
__host__ __device__ __forceinline__ int hz_rcode(int h) { return (h >> HZ_R_SHIFT) & HZ_CODE_MASK; }
__host__ __device__ __forceinline__ int hz_war(int h) { return (h >> HZ_WAR_SHIFT) & 63; }

// Launch geometry of the recurrence (depends only on the shape).
struct RecPlan {
    int dch;      // 16-byte chunks of a row per warp (its d-range)
    int nsplit;   // d-ranges per chain
    int spt;      // slot positions per lane per token
    int la;       // hazard window in tokens (prefetches in flight ahead of the processed token)
    int kmax;     // max(k_write, k_read)
    int w;        // warps per CTA interleaving the tokens of one (chain, d-range); 0: one token
                  // per chain (T == 1), one warp per (chain, d-range), no look-ahead
    int p;        // prefetch depth of each interleaving warp, in its own tokens
};
RecPlan rec_plan(int dtype, int B, int H, int T, int dv, int kw, int kr);
// Scratch of the recurrence: the hazard table [B, H, T, max(kw, kr)] int32.
size_t rec_workspace_bytes(int B, int H, int T, int kw, int kr);
// Runs the hazard pass, then the recurrence.  hz_ws: rec_workspace_bytes() of scratch.
// firstw (lazy initial memory, with a.M0 set): [B*H, N] first writer of each slot in this
// call (-1: written by an earlier call; INT_MAX: not written), see k_lazy.cu.
// mem_ready: when given, the stream waits on it after the hazard pass, before the recurrence
// (the hazard pass reads only the lists, so it can run while mem is still being written).
cudaError_t launch_recur(int dtype, const RecArgs& a, int32_t* hz_ws, cudaStream_t stream,
                         const int32_t* firstw = nullptr, cudaEvent_t mem_ready = nullptr);

// Backward of the recurrence with in-place undo (k_recur_bwd.cu).  a.mem holds M_T on entry and
// M_0 on return; dM ([B, H, N, dv] fp32, zero on entry) receives dL/dM_0 per chain.  kind 0:
// the log is `undo` (stored rows); kind 1 / 2: fp8 / int4 codes with one float32 scale per row.
cudaError_t launch_recur_backward(int dtype, const RecArgs& a, int kind, const void* undo, const void* codes,
                                  const float* scales, const void* dy, float* dv, float* dalpha, float* dbeta,
                                  float* dw_w, float* dw_r, float* dM, cudaStream_t stream);
// Quantised snapshot of an undo log of `rows` rows of dv storage elements (kind 1: fp8 e4m3 codes,
// dv bytes per row; kind 2: int4 codes, dv / 2 bytes per row), one float32 scale per row.
cudaError_t launch_undo_quantize(int dtype, int kind, const void* undo, int64_t rows, int dv, void* codes,
                                 float* scales, cudaStream_t stream);

// Chunkwise (WY) form of the recurrence (k_chunk.cu), chunks of C <= 32 tokens; d_v <= 256.
cudaError_t launch_recur_chunkwise(int dtype, const RecArgs& a, int C, cudaStream_t stream);
size_t chunk_smem_bytes(int C, int kw, int kr, int dv);

// ---------------------------------------------------------------- K-LAZY (k_lazy.cu)
// firstw from the touched bitmap [chains, ceil(N/32)], then the first writer of every slot.
cudaError_t launch_lazy_prepare(const uint32_t* touched, int32_t* firstw, const int32_t* idx_w, int64_t chains, int T,
                                int kw, int64_t N, cudaStream_t stream);
// touched bitmap from firstw (after launch_lazy_prepare).
cudaError_t launch_lazy_bitmap(const int32_t* firstw, uint32_t* touched, int64_t chains, int64_t N, cudaStream_t stream);
// Gate preparation and output epilogue (k_gates.cu).  dtype 0 = fp32, 1 = bf16 storage.
cudaError_t launch_gates(int dtype, const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A,
                         void* alpha, void* beta, int B, int T, int H, int d, cudaStream_t stream);
// Tensor-core forms (k_gemm.cu, bf16 only).  Gates: alpha, beta as launch_gates, for H in
// {16, 32} and d % 8 == 0.  Head mix: out [M, N] = z [M, K] W_o^T with W_o [N, K], N % 32 == 0,
// K % 8 == 0.  A bounded wait that runs out sets ERR_TIMEOUT in err.
bool gates_tc_supported(int dtype, int H, int d);
cudaError_t launch_gates_tc(const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A,
                            void* alpha, void* beta, int B, int T, int H, int d, int* err, cudaStream_t stream);
cudaError_t launch_head_mix(const void* z, const void* W_o, void* out, int64_t M, int N, int K, int* err,
                            cudaStream_t stream);
cudaError_t launch_norm_gate(int dtype, const void* y, const void* g, const float* gamma, float eps, void* z, int B, int H,
                             int T, int dv, cudaStream_t stream);
// Access diagnostics (k_stats.cu): bits = 2 * chains * ceil(N/32) words of scratch; out =
// 4 + kw + kr float64 sums (see sdm_access_stats).
cudaError_t launch_access_stats(const int32_t* idx_w, const float* w_w, const int32_t* idx_r, const float* w_r,
                                int64_t chains, int T, int kw, int kr, int64_t N, uint32_t* bits, double* out,
                                cudaStream_t stream);
// mem rows of untouched slots = M0 rows (rowbytes a multiple of 16).
cudaError_t launch_materialize(const void* M0, const uint32_t* touched, void* mem, int64_t chains, int H, int64_t N,
                               int64_t rowbytes, cudaStream_t stream);

// Error reporting and the checks of sdm_recur (minus its workspace), for entry points
// in other translation units (sdm_api.cu).
sdm_status api_error(sdm_status st, const char* msg);
sdm_status api_ok();
sdm_status recur_args(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                      const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                      void* mem, void* y, RecArgs* r, bool* empty);

}  // namespace sdm
