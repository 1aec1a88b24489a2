// K-ADDR scores on the 5th-generation tensor cores (bf16 storage, PROJECTED addressing).
//
// The half-scores s = P x (Sec. 3.1 item 1) of 128 tokens x one column chunk (<= 512
// columns of one half) form a dense [128 x d_k] x [d_k x NP] contraction: TMA stages the x
// tile and the chunk's rows of P in shared memory (128-byte swizzle, K-major), one thread
// issues tcgen05.mma (M = 128, N <= 256 per instruction, K = 16 per step, bf16 inputs, fp32
// accumulation in TMEM), and each of the 128 threads then owns one token's TMEM row.
//
// Per-token top-L selection of the chunk (L = k + 4; the finalize kernel certifies it), all
// branch-free so a warp's 32 tokens run in lockstep; the passes over TMEM are loops over
// 32-column blocks (compact code: the kernel is instruction-fetch bound when unrolled):
//   1. the two largest scores of each of the 32 column classes mod 32;
//   2. theta0 = L-th largest of those 64 values (bitonic network) -- a provable lower bound
//      on the L-th largest score, since >= L distinct columns are >= it;
//   3. survivors (score >= theta0) compacted into a per-thread shared-memory buffer with
//      predicated stores (the P buffer is free once the MMA has completed);
//   4. survivors sorted by a 64-entry bitonic network; the first L go to the workspace.
// More than 64 survivors: the warp repeats with the L-th largest of the first 64 survivors
// as threshold (still a lower bound); after three rounds (heavy ties) an exact insertion
// scan over the chunk decides.
#include "sdm_internal.h"
#include "tc_common.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

namespace sdm {

namespace {

using namespace tc;

constexpr int MM_THREADS = 128;      // = tokens per CTA = TMEM lanes
constexpr int MM_NB = 256;           // columns per MMA instruction
constexpr int MM_BUF = 64;           // survivor slots per thread

// Bytes of the region that holds the chunk's rows of P and, once the MMA has completed,
// the survivor buffers (values and indices, MM_BUF slots per thread).
__host__ __device__ constexpr uint32_t mma_region_bytes(int atoms, int cols) {
    return static_cast<uint32_t>(atoms) * cols * 128 > 2u * MM_BUF * MM_THREADS * 4
               ? static_cast<uint32_t>(atoms) * cols * 128
               : 2u * MM_BUF * MM_THREADS * 4;
}

// Bitonic sort, descending by value (ties in any order); values only / value-index pairs.
template <int N>
__device__ __forceinline__ void bitonic_desc(float (&v)[N]) {
#pragma unroll
    for (int size = 2; size <= N; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
            for (int i = 0; i < N; ++i) {
                const int j = i ^ stride;
                if (j > i) {
                    const float a = v[i], b = v[j];
                    if ((i & size) == 0) { v[i] = fmaxf(a, b); v[j] = fminf(a, b); }
                    else { v[i] = fminf(a, b); v[j] = fmaxf(a, b); }
                }
            }
}
template <int N>
__device__ __forceinline__ void bitonic_desc(float (&v)[N], int (&ix)[N]) {
#pragma unroll
    for (int size = 2; size <= N; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
            for (int i = 0; i < N; ++i) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool up = (i & size) == 0;
                    const bool sw = up ? (v[i] < v[j]) : (v[i] > v[j]);
                    const float a = v[i];
                    const int ia = ix[i];
                    v[i] = sw ? v[j] : a;   ix[i] = sw ? ix[j] : ia;
                    v[j] = sw ? a : v[j];   ix[j] = sw ? ia : ix[j];
                }
            }
}

}  // namespace

struct MmaLaunch {
    int B, H, T, dk, S;
    int bt, bb, ntt;            // token box: bt tokens x bb sequences (bt * bb <= 128); t-tiles
    int pb;                     // P box height (rows), <= 256 and <= 2S
    int ncc, cw;                // chunks per half, columns per chunk
    int L;                      // list length kept per chunk
    int atoms;                  // ceil(dk / 64)
    float* part_v;
    int* part_i;
    int* err;
    float* raw;                 // test hook: the raw fp32 scores [2H][B*T][2S] instead of the lists
};

// COLS: TMEM columns (fp32 accumulators) = maximum chunk width (512: one CTA per SM;
// 256: two CTAs per SM).
template <int COLS>
__global__ void __launch_bounds__(MM_THREADS, 1) k_addr_mma(const __grid_constant__ CUtensorMap tx_q,
                                                            const __grid_constant__ CUtensorMap tx_k,
                                                            const __grid_constant__ CUtensorMap tp_q,
                                                            const __grid_constant__ CUtensorMap tp_k, const MmaLaunch a) {
    extern __shared__ unsigned char sm_raw[];
    // 1024-byte aligned operand region (the 128-byte swizzle repeats every 8 rows = 1024 B)
    const uint32_t raw = smem_u32(sm_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char* sm = sm_raw + (base - raw);
    const uint32_t sA = base;                                   // [atoms][128 rows][128 B]
    const uint32_t sB = sA + a.atoms * 128 * 128;                // [atoms][COLS rows][128 B]; survivors later
    const uint32_t sBar = sB + mma_region_bytes(a.atoms, COLS);  // 3 mbarriers + TMEM address
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + (sBar - base) + 32);
    float* buf_v = reinterpret_cast<float*>(sm + (sB - base));                       // [MM_BUF][128]
    int* buf_i = reinterpret_cast<int*>(sm + (sB - base) + MM_BUF * MM_THREADS * 4);  // [MM_BUF][128]

    const int tid = threadIdx.x, warp = tid >> 5;
    const int side = blockIdx.z / a.H, h = blockIdx.z % a.H;
    const int chunk = blockIdx.y;
    const int hf = chunk / a.ncc, cc = chunk % a.ncc;
    const int c0 = cc * a.cw;
    const int np = min(a.S, c0 + a.cw) - c0;                     // valid columns of this chunk
    const int npad = (np + 15) & ~15;
    const int ti = blockIdx.x % a.ntt, bi = blockIdx.x / a.ntt;
    const int t0 = ti * a.bt, b0 = bi * a.bb;
    const CUtensorMap* tx = side ? &tx_k : &tx_q;
    const CUtensorMap* tp = side ? &tp_k : &tp_q;
    const uint32_t bar_x = sBar, bar_p = sBar + 8, bar_mma = sBar + 16;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)), "r"(COLS) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    if (tid == 0) {
        mbar_init(bar_x, 1);
        mbar_init(bar_p, 1);
        mbar_init(bar_mma, 1);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    bool ok = true;
    if (tid == 0) {
        // x tile: rows = (b0 .. b0+bb-1) x (t0 .. t0+bt-1) of head h; P rows of the chunk
        mbar_expect_tx(bar_x, a.atoms * a.bt * a.bb * 128);
        for (int at = 0; at < a.atoms; ++at) tma_load_4d(sA + at * 128 * 128, tx, at * 64, t0, h, b0, bar_x);
        const int nblk = (npad + MM_NB - 1) / MM_NB;
        mbar_expect_tx(bar_p, a.atoms * nblk * a.pb * 128);
        for (int at = 0; at < a.atoms; ++at)
            for (int nb = 0; nb < nblk; ++nb)
                tma_load_3d(sB + at * COLS * 128 + nb * MM_NB * 128, tp, at * 64, hf * a.S + c0 + nb * MM_NB, h, bar_p);
        ok = mbar_wait(bar_x, 0) && mbar_wait(bar_p, 0);
        if (ok) {
            asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
            for (int nb = 0; nb < nblk; ++nb) {
                const int n = min(MM_NB, npad - nb * MM_NB);
                const uint32_t idesc = mma_idesc(n);
                for (int ks = 0; ks < a.atoms * 4; ++ks) {
                    const uint32_t aoff = (ks >> 2) * 128 * 128 + (ks & 3) * 32;
                    const uint32_t boff = (ks >> 2) * COLS * 128 + nb * MM_NB * 128 + (ks & 3) * 32;
                    mma_bf16(tmem + nb * MM_NB, sw128_desc(sA + aoff), sw128_desc(sB + boff), idesc, ks > 0 ? 1u : 0u);
                }
            }
            mma_commit(bar_mma);
        }
    }
    ok = __syncthreads_and(ok);
    if (ok) ok = mbar_wait(bar_mma, 0);
    ok = __syncthreads_and(ok);
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");

    const int L = a.L;
    const int64_t BT = static_cast<int64_t>(a.B) * a.T;
    const int b = b0 + tid / a.bt, t = t0 + tid % a.bt;
    const bool valid = ok && b < a.B && t < a.T;
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const int nblk32 = npad / 32 + ((npad & 31) ? 1 : 0);   // 32-column blocks with columns

    if (a.raw != nullptr) {
        // test hook: the accumulators themselves, one token row per thread, no selection
        float* dst = a.raw + (static_cast<int64_t>(blockIdx.z) * BT + static_cast<int64_t>(b) * a.T + t) * (2 * a.S) + hf * a.S + c0;
#pragma unroll 1
        for (int cb = 0; cb < nblk32; ++cb) {
            float v[32];
            tmem_ld32(trow + cb * 32, v);                        // warp-collective: every lane loads
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (valid && cb * 32 + j < np) dst[cb * 32 + j] = v[j];
        }
        if (!ok && tid == 0) flag_error(a.err, ERR_TIMEOUT);
        asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
        __syncthreads();
        if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(COLS) : "memory");
        return;
    }

    // 1-2. top-2 of each column class mod 32; threshold = L-th largest of those 64 values
    // (>= L distinct columns reach it, so it is a lower bound on the L-th largest score)
    float theta = -INFINITY;
    if (ok) {
        float m1[32], m2[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) { m1[i] = -INFINITY; m2[i] = -INFINITY; }
#pragma unroll 1
        for (int cb = 0; cb < nblk32; ++cb) {
            float v[32];
            tmem_ld32(trow + cb * 32, v);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const float x = cb * 32 + j < np ? v[j] : -INFINITY;
                m2[j] = fmaxf(m2[j], fminf(m1[j], x));
                m1[j] = fmaxf(m1[j], x);
            }
        }
        if (np >= L) {
            float g64[64];
#pragma unroll
            for (int i = 0; i < 32; ++i) { g64[i] = m1[i]; g64[32 + i] = m2[i]; }
            bitonic_desc<64>(g64);
            float th = g64[0];
#pragma unroll
            for (int i = 1; i < 64; ++i) th = (i == L - 1) ? g64[i] : th;
            theta = th;
        }
    }

    // 3-4. compaction of survivors, then sort; overflowing warps repeat with the L-th largest
    // survivor kept so far as threshold (still a lower bound on the L-th largest score)
    float outv[MM_BUF];
    int outi[MM_BUF];
    bool exact_fallback = false;
    for (int round = 0; round < 3; ++round) {
        int cnt = 0;
        if (ok) {
#pragma unroll 1
            for (int cb = 0; cb < nblk32; ++cb) {
                float v[32];
                tmem_ld32(trow + cb * 32, v);
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const int col = cb * 32 + j;
                    const bool keep = col < np && v[j] >= theta;
                    if (keep && cnt < MM_BUF) {
                        buf_v[cnt * MM_THREADS + tid] = v[j];
                        buf_i[cnt * MM_THREADS + tid] = c0 + col;
                    }
                    cnt += keep ? 1 : 0;
                }
            }
        }
#pragma unroll
        for (int i = 0; i < MM_BUF; ++i) {
            outv[i] = i < cnt ? buf_v[i * MM_THREADS + tid] : -INFINITY;
            outi[i] = i < cnt ? buf_i[i * MM_THREADS + tid] : 0x7fffffff;
        }
        bitonic_desc<MM_BUF>(outv, outi);
        const bool overflow = cnt > MM_BUF;
        if (!__any_sync(0xffffffffu, overflow)) break;
        if ((tid & 31) == 0) stat_add(a.err, STAT_SELECT_RETRY);
        if (overflow) {
            float th = outv[0];
#pragma unroll
            for (int i = 1; i < MM_BUF; ++i) th = (i == L - 1) ? outv[i] : th;
            if (round == 2) exact_fallback = true;
            theta = th;
        }
    }
    if (__any_sync(0xffffffffu, exact_fallback)) {
        // heavy ties: exact top-L by insertion over the chunk (rare, slow).  Every lane of the
        // warp runs the TMEM loads (they are warp-collective); only flagged lanes insert.
        float lv[MM_BUF];
        int li[MM_BUF];
        for (int i = 0; i < MM_BUF; ++i) { lv[i] = -INFINITY; li[i] = 0x7fffffff; }
        for (int col = 0; col < np; ++col) {
            uint32_t xb;
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];\n" : "=r"(xb) : "r"(trow + col));
            asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
            const float x = __uint_as_float(xb);
            if (exact_fallback && x > lv[L - 1]) {
                int p = L - 1;
                while (p > 0 && x > lv[p - 1]) { lv[p] = lv[p - 1]; li[p] = li[p - 1]; --p; }
                lv[p] = x; li[p] = c0 + col;
            }
        }
        if (exact_fallback) {
            for (int i = 0; i < MM_BUF; ++i) { outv[i] = lv[i]; outi[i] = li[i]; }
        }
    }
    if (valid) {   // the token's L entries are contiguous (L % 4 == 0): 16-byte stores
        const int64_t u = static_cast<int64_t>(b) * a.T + t;
        const int64_t lbase = ((static_cast<int64_t>(blockIdx.z) * (2 * a.ncc) + chunk) * BT + u) * L;
        float4* pv = reinterpret_cast<float4*>(a.part_v + lbase);
        int4* pi = reinterpret_cast<int4*>(a.part_i + lbase);
#pragma unroll
        for (int i = 0; i < MM_BUF; i += 4)
            if (i < L) {
                pv[i / 4] = make_float4(outv[i], outv[i + 1], outv[i + 2], outv[i + 3]);
                pi[i / 4] = make_int4(outi[i], outi[i + 1], outi[i + 2], outi[i + 3]);
            }
    }
    if (!ok && tid == 0) flag_error(a.err, ERR_TIMEOUT);

    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(COLS) : "memory");
}

// ------------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------------
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

}  // namespace

bool mma_path_supported(int dtype, int direct, int dk, int S, int kmax) {
    return dtype == 1 && !direct && (dk == 64 || dk == 128) && kmax <= 32 && S >= 16;
}

// A CTA allocates `cols` TMEM columns of the SM's 512: a 512-column CTA asks for enough
// shared memory that no second CTA is resident beside it.
size_t mma_smem_bytes(int dk, int cols) {
    const int atoms = (dk + 63) / 64;
    const size_t need = 1024 + static_cast<size_t>(atoms) * 128 * 128 + mma_region_bytes(atoms, cols) + 64;
    const size_t one_per_sm = 120 * 1024;
    return cols >= 512 && need < one_per_sm ? one_per_sm : need;
}

cudaError_t launch_address_mma(const AddrPlan& plan, const AddrArgs& aa, cudaStream_t stream) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    MmaLaunch a{};
    a.B = aa.B; a.H = aa.H; a.T = aa.T; a.dk = aa.dk; a.S = aa.S;
    a.bt = 1;
    while (a.bt * 2 <= aa.T && a.bt < 128) a.bt *= 2;     // largest power of two <= min(T, 128)
    a.bb = 128 / a.bt;
    if (a.bb > aa.B) a.bb = aa.B;                          // boxes never exceed the tensor
    a.ntt = (aa.T + a.bt - 1) / a.bt;
    const int nbt = (aa.B + a.bb - 1) / a.bb;
    a.pb = 2 * aa.S < MM_NB ? 2 * aa.S : MM_NB;
    a.ncc = plan.ncc;
    a.cw = plan.cw;
    a.L = plan.L;
    a.atoms = (aa.dk + 63) / 64;
    a.part_v = aa.part_v;
    a.part_i = aa.part_i;
    a.err = aa.err;
    a.raw = aa.raw;

    CUtensorMap maps[4];
    for (int s = 0; s < 2; ++s) {
        // x: dims {dk, T, H, B}; box {64, bt, 1, bb}
        cuuint64_t gdim[4] = {static_cast<cuuint64_t>(aa.dk), static_cast<cuuint64_t>(aa.T), static_cast<cuuint64_t>(aa.H),
                              static_cast<cuuint64_t>(aa.B)};
        cuuint64_t gstr[3] = {static_cast<cuuint64_t>(aa.dk) * 2, static_cast<cuuint64_t>(aa.dk) * 2 * aa.T,
                              static_cast<cuuint64_t>(aa.dk) * 2 * aa.T * aa.H};
        cuuint32_t box[4] = {64, static_cast<cuuint32_t>(a.bt), 1, static_cast<cuuint32_t>(a.bb)};
        cuuint32_t es[4] = {1, 1, 1, 1};
        CUresult r = enc(&maps[s], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(aa.X[s]), gdim, gstr, box, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
        // P: dims {dk, 2S, H}; box {64, 256, 1}
        cuuint64_t pdim[3] = {static_cast<cuuint64_t>(aa.dk), static_cast<cuuint64_t>(2 * aa.S), static_cast<cuuint64_t>(aa.H)};
        cuuint64_t pstr[2] = {static_cast<cuuint64_t>(aa.dk) * 2, static_cast<cuuint64_t>(aa.dk) * 2 * 2 * aa.S};
        cuuint32_t pbox[3] = {64, static_cast<cuuint32_t>(a.pb), 1};
        cuuint32_t pes[3] = {1, 1, 1};
        r = enc(&maps[2 + s], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(aa.P[s]), pdim, pstr, pbox, pes,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    dim3 grid(static_cast<unsigned>(a.ntt * nbt), 2 * plan.ncc, 2 * aa.H);
    cudaError_t e = cudaSuccess;
    if (plan.cw <= 256) {
        const size_t smem = mma_smem_bytes(aa.dk, 256);
        e = cudaFuncSetAttribute(k_addr_mma<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_addr_mma<256><<<grid, MM_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], maps[3], a);
    } else {
        const size_t smem = mma_smem_bytes(aa.dk, 512);
        e = cudaFuncSetAttribute(k_addr_mma<512>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        k_addr_mma<512><<<grid, MM_THREADS, smem, stream>>>(maps[0], maps[1], maps[2], maps[3], a);
    }
    return cudaGetLastError();
}

}  // namespace sdm
