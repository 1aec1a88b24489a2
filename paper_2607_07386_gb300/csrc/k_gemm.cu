// Dense contractions around the SDM path on the 5th-generation tensor cores (bf16 operands,
// fp32 accumulation in TMEM):
//
//   k_gates_tc    the gate projections of every token (Sec. 3.1, after Eq. sdm-write):
//                   [s_a | s_b] = x [W_a; W_b]^T,  x: [B*T, d_model],  N = 2H columns,
//                 with the gate nonlinearities as the epilogue:
//                   alpha = exp(-A softplus(s_a + b_dt)),  beta = sigmoid(s_b).
//   k_head_mix    the head-mixing projection o = z W_o^T ("Norm, Gating, and Head Mixing"),
//                 z: [B*T, H*d_v] (the token-major output of sdm_norm_gate), W_o: [d_model, H*d_v].
//
// Both are one kernel shape: a CTA owns 128 rows (TMEM lanes) x BN columns; TMA streams
// K-blocks of 64 bf16 (one 128-byte swizzle atom) of both operands through an S-stage ring of
// shared memory; one thread issues the loads and the tcgen05.mma (M = 128, N = BN, K = 16 per
// instruction) and releases a stage with tcgen05.commit once the MMAs that read it are done;
// after the last K-block the four warps read their 32 lanes of the accumulator with tcgen05.ld
// and run the epilogue.  Every wait is bounded; a wait that runs out sets the timeout bit of the
// status word and the CTA skips its epilogue.
#include "sdm_internal.h"
#include "tc_common.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

namespace sdm {

namespace {

using namespace tc;

constexpr int GM_THREADS = 128;      // = rows per CTA = TMEM lanes
constexpr int GM_BK = 64;            // K per stage: one 128-byte swizzle atom of bf16

__host__ __device__ constexpr uint32_t gm_stage_bytes(int bn) { return (128u + static_cast<uint32_t>(bn)) * 128u; }
__host__ __device__ constexpr uint32_t gm_smem_bytes(int bn, int stages) {
    return 1024u + gm_stage_bytes(bn) * stages + 256u;      // alignment slack, ring, barriers
}

PFN_cuTensorMapEncodeTiled_v12000 gm_encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// 2-D bf16 tensor map of a row-major [rows, cols] matrix, box {64 columns, box_rows rows},
// 128-byte swizzle (the K-major operand layout of the MMA descriptors).
bool gm_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = gm_encode_fn();
    if (!enc) return false;
    cuuint64_t dim[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t str[1] = {static_cast<cuuint64_t>(cols) * 2};
    cuuint32_t box[2] = {GM_BK, static_cast<cuuint32_t>(box_rows)};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dim, str, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The pipelined main loop, run by thread 0: K-blocks of both operands into the ring, four
// MMAs per K-block into the accumulator at `tmem`, then a commit to `done`.  B comes from one
// map (rows n0 .. n0 + BN) or, with tb2, from two maps of BN / 2 rows each (stacked).
template <int BN, int S>
__device__ bool gm_mainloop(const CUtensorMap* ta, const CUtensorMap* tb, const CUtensorMap* tb2, int m0, int n0,
                            int nkb, uint32_t ring, uint32_t bars, uint32_t tmem) {
    const uint32_t full = bars, empty = bars + 8 * S, done = bars + 16 * S;
    const uint32_t stage = gm_stage_bytes(BN);
    const uint32_t idesc = mma_idesc(BN);
    auto load = [&](int kb, int s) {
        const uint32_t a = ring + s * stage, b = a + 128 * 128;
        mbar_expect_tx(full + 8 * s, stage);
        tma_load_2d(a, ta, kb * GM_BK, m0, full + 8 * s);
        if (tb2 == nullptr) {
            tma_load_2d(b, tb, kb * GM_BK, n0, full + 8 * s);
        } else {
            tma_load_2d(b, tb, kb * GM_BK, 0, full + 8 * s);
            tma_load_2d(b + (BN / 2) * 128, tb2, kb * GM_BK, 0, full + 8 * s);
        }
    };
    bool ok = true;
    const int pre = nkb < S ? nkb : S;
    for (int kb = 0; kb < pre; ++kb) load(kb, kb);
    for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % S;
        const uint32_t ph = static_cast<uint32_t>(kb / S) & 1u;
        if (!mbar_wait(full + 8 * s, ph)) { ok = false; break; }
        asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
        const uint32_t a = ring + s * stage, b = a + 128 * 128;
#pragma unroll
        for (int kk = 0; kk < GM_BK / 16; ++kk)
            mma_bf16(tmem, sw128_desc(a + kk * 32), sw128_desc(b + kk * 32), idesc, (kb | kk) != 0 ? 1u : 0u);
        mma_commit(empty + 8 * s);             // arrives once these MMAs have read the stage
        if (kb + S < nkb) {
            if (!mbar_wait(empty + 8 * s, ph)) { ok = false; break; }
            load(kb + S, s);
        }
    }
    mma_commit(done);                          // every MMA issued above has completed
    return ok;
}

// Shared set-up of both kernels: ring aligned to 1024 bytes, barriers, TMEM allocation.
struct GmCta {
    uint32_t ring, bars, tmem;
};

template <int BN, int S>
__device__ GmCta gm_setup(unsigned char* sm_raw) {
    const uint32_t raw = smem_u32(sm_raw);
    const uint32_t ring = (raw + 1023u) & ~1023u;
    const uint32_t bars = ring + gm_stage_bytes(BN) * S;       // full[S], empty[S], done, TMEM address
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm_raw + (bars - raw) + 16 * S + 8);
    const int tid = threadIdx.x;
    if (tid < 32) {
        constexpr uint32_t cols = BN < 32 ? 32 : BN;
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)), "r"(cols) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(bars + 8 * s, 1);
            mbar_init(bars + 8 * S + 8 * s, 1);
        }
        mbar_init(bars + 16 * S, 1);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    return GmCta{ring, bars, *tmem_slot};
}

template <int BN>
__device__ void gm_teardown(uint32_t tmem) {
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    constexpr uint32_t cols = BN < 32 ? 32 : BN;
    if (threadIdx.x < 32) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(cols) : "memory");
}

// Main loop, then every thread waits for the accumulator (bounded).
template <int BN, int S>
__device__ bool gm_run(const GmCta& c, const CUtensorMap* ta, const CUtensorMap* tb, const CUtensorMap* tb2, int m0,
                       int n0, int nkb) {
    bool ok = true;
    if (threadIdx.x == 0) ok = gm_mainloop<BN, S>(ta, tb, tb2, m0, n0, nkb, c.ring, c.bars, c.tmem);
    ok = __syncthreads_and(ok);
    if (ok) ok = mbar_wait(c.bars + 16 * S, 0);
    ok = __syncthreads_and(ok);
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    return ok;
}

// ------------------------------------------------------------------------------------------
// Gates: BN = 2H columns (32 or 64), rows = tokens.
// ------------------------------------------------------------------------------------------
constexpr int GATE_STAGES = 4;

template <int BN>
__global__ void __launch_bounds__(GM_THREADS) k_gates_tc(const __grid_constant__ CUtensorMap tx,
                                                         const __grid_constant__ CUtensorMap twa,
                                                         const __grid_constant__ CUtensorMap twb,
                                                         const float* __restrict__ b_dt, const float* __restrict__ A,
                                                         __nv_bfloat16* __restrict__ alpha, __nv_bfloat16* __restrict__ beta,
                                                         int64_t tokens, int T, int d, int* err) {
    constexpr int H = BN / 2;
    extern __shared__ unsigned char sm_raw[];
    const GmCta c = gm_setup<BN, GATE_STAGES>(sm_raw);
    const int m0 = blockIdx.x * 128;
    const int nkb = (d + GM_BK - 1) / GM_BK;
    const bool ok = gm_run<BN, GATE_STAGES>(c, &tx, &twa, &twb, m0, 0, nkb);
    const int warp = threadIdx.x >> 5;
    const int64_t u = m0 + threadIdx.x;                   // this thread's token row
    if (ok) {
        const uint32_t trow = c.tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll
        for (int cb = 0; cb < BN / 32; ++cb) {
            float v[32];
            tmem_ld32(trow + cb * 32, v);                  // warp-collective
            if (u < tokens) {
                const int64_t b = u / T, t = u - b * T;
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int j = cb * 32 + i;
                    if (j < H) {
                        const float za = v[i] + __ldg(b_dt + j);
                        const float sp = za > 20.f ? za : log1pf(expf(za));     // softplus
                        alpha[(b * H + j) * T + t] = __float2bfloat16_rn(expf(-__ldg(A + j) * sp));
                    } else {
                        beta[(b * H + (j - H)) * T + t] = __float2bfloat16_rn(1.f / (1.f + expf(-v[i])));
                    }
                }
            }
        }
    } else if (threadIdx.x == 0) {
        flag_error(err, ERR_TIMEOUT);
    }
    gm_teardown<BN>(c.tmem);
}

// ------------------------------------------------------------------------------------------
// Head mix: BN = 256 output columns per CTA, out row-major [M, N] bf16.
// ------------------------------------------------------------------------------------------
constexpr int MIX_BN = 256;
constexpr int MIX_STAGES = 4;

__global__ void __launch_bounds__(GM_THREADS, 1) k_head_mix(const __grid_constant__ CUtensorMap tz,
                                                            const __grid_constant__ CUtensorMap tw,
                                                            __nv_bfloat16* __restrict__ out, int64_t M, int N, int K,
                                                            int* err) {
    extern __shared__ unsigned char sm_raw[];
    const GmCta c = gm_setup<MIX_BN, MIX_STAGES>(sm_raw);
    const int ntn = (N + MIX_BN - 1) / MIX_BN;
    const int m0 = static_cast<int>(blockIdx.x / ntn) * 128, n0 = static_cast<int>(blockIdx.x % ntn) * MIX_BN;
    const bool ok = gm_run<MIX_BN, MIX_STAGES>(c, &tz, &tw, nullptr, m0, n0, (K + GM_BK - 1) / GM_BK);
    const int warp = threadIdx.x >> 5;
    const int64_t r = m0 + threadIdx.x;
    if (ok) {
        const uint32_t trow = c.tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll 1
        for (int cb = 0; cb < MIX_BN / 32; ++cb) {
            float v[32];
            tmem_ld32(trow + cb * 32, v);                  // warp-collective
            const int n = n0 + cb * 32;
            if (r < M && n < N) {                          // N % 32 == 0: whole 32-column blocks
                uint4* dst = reinterpret_cast<uint4*>(out + r * N + n);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        __nv_bfloat162 p = __floats2bfloat162_rn(v[q * 8 + 2 * e], v[q * 8 + 2 * e + 1]);
                        w[e] = *reinterpret_cast<uint32_t*>(&p);
                    }
                    dst[q] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
        }
    } else if (threadIdx.x == 0) {
        flag_error(err, ERR_TIMEOUT);
    }
    gm_teardown<MIX_BN>(c.tmem);
}

}  // namespace

bool gates_tc_supported(int dtype, int H, int d) {
    return dtype == 1 && (H == 16 || H == 32) && d % 8 == 0 && d > 0;
}

cudaError_t launch_gates_tc(const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A,
                            void* alpha, void* beta, int B, int T, int H, int d, int* err, cudaStream_t stream) {
    const int64_t tokens = static_cast<int64_t>(B) * T;
    CUtensorMap maps[3];
    if (!gm_map(&maps[0], x, tokens, d, 128) || !gm_map(&maps[1], W_a, H, d, H) || !gm_map(&maps[2], W_b, H, d, H))
        return cudaErrorInvalidValue;
    const unsigned grid = static_cast<unsigned>((tokens + 127) / 128);
    auto* al = static_cast<__nv_bfloat16*>(alpha);
    auto* be = static_cast<__nv_bfloat16*>(beta);
    cudaError_t e;
    if (H == 16) {
        const size_t smem = gm_smem_bytes(32, GATE_STAGES);
        e = cudaFuncSetAttribute(k_gates_tc<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_gates_tc<32><<<grid, GM_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], b_dt, A, al, be, tokens, T, d, err);
    } else {
        const size_t smem = gm_smem_bytes(64, GATE_STAGES);
        e = cudaFuncSetAttribute(k_gates_tc<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_gates_tc<64><<<grid, GM_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], b_dt, A, al, be, tokens, T, d, err);
    }
    return cudaGetLastError();
}

cudaError_t launch_head_mix(const void* z, const void* W_o, void* out, int64_t M, int N, int K, int* err,
                            cudaStream_t stream) {
    CUtensorMap maps[2];
    if (!gm_map(&maps[0], z, M, K, 128) || !gm_map(&maps[1], W_o, N, K, MIX_BN)) return cudaErrorInvalidValue;
    const int64_t tiles = ((M + 127) / 128) * ((N + MIX_BN - 1) / MIX_BN);
    const size_t smem = gm_smem_bytes(MIX_BN, MIX_STAGES);
    cudaError_t e = cudaFuncSetAttribute(k_head_mix, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    k_head_mix<<<static_cast<unsigned>(tiles), GM_THREADS, smem, stream>>>(maps[0], maps[1],
                                                                           static_cast<__nv_bfloat16*>(out), M, N, K, err);
    return cudaGetLastError();
}

}  // namespace sdm
