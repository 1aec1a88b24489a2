// The steps on either side of the SDM path in a layer (Sec. 3.1):
//
//   k_gates      per-head gates of every token from the layer input x_t (after Eq. sdm-write):
//                  alpha_t = exp(-A softplus(W_a x_t + b_dt)),  beta_t = sigmoid(W_b x_t)
//                One warp per token: lanes split x_t into 16-byte vectors, every lane
//                accumulates all 2H dot products against W_a and W_b (staged in shared memory
//                when they fit), warp reductions finish them, and lane j writes gate j.  x is
//                read once: 2H * d FMAs per token, B*T*d*elem bytes of HBM.
//   k_norm_gate  z = g (.) RMSNorm(y) per head ("Norm, Gating, and Head Mixing"), with the
//                RMSNorm scale gamma: z = g * gamma * y / sqrt(mean(y^2) + eps).  One warp per
//                (b, h, t) row; z is written token-major [B, T, H, d_v], the layout in which the
//                head-mixing projection W_o is one plain GEMM.  HBM-bound: y and g read once, z
//                written once.
#include "sdm_internal.h"

namespace sdm {

constexpr int GT_THREADS = 256;        // k_norm_gate
constexpr int GG_THREADS = 512;        // k_gates: 16 warps share one copy of W_a, W_b per SM
constexpr size_t GT_SMEM_MAX = 200 * 1024;

template <class D> __device__ __forceinline__ void store_elem(void* base, int64_t i, float v);
template <> __device__ __forceinline__ void store_elem<F32>(void* base, int64_t i, float v) {
    reinterpret_cast<float*>(base)[i] = v;
}
template <> __device__ __forceinline__ void store_elem<BF16>(void* base, int64_t i, float v) {
    reinterpret_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(v);
}

// 8-byte chunks (4 bf16 or 2 fp32) of a row.
template <class D> struct Chunk8;
template <> struct Chunk8<F32> {
    static constexpr int E = 2;
    __device__ static void unpack(uint2 u, float* f) { f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y); }
    __device__ static uint2 pack(const float* f) { return make_uint2(__float_as_uint(f[0]), __float_as_uint(f[1])); }
};
template <> struct Chunk8<BF16> {
    static constexpr int E = 4;
    __device__ static void unpack(uint2 u, float* f) {
        f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xffff0000u);
        f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xffff0000u);
    }
    __device__ static uint2 pack(const float* f) {
        __nv_bfloat162 a = __floats2bfloat162_rn(f[0], f[1]), b = __floats2bfloat162_rn(f[2], f[3]);
        return make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
    }
};

// NH >= 2H accumulators per lane.
template <class D, int NH>
__global__ void __launch_bounds__(GG_THREADS) k_gates(const void* __restrict__ x, const void* __restrict__ W_a,
                                                      const void* __restrict__ W_b, const float* __restrict__ b_dt,
                                                      const float* __restrict__ A, void* __restrict__ alpha,
                                                      void* __restrict__ beta, int64_t tokens, int T, int H, int d,
                                                      int use_smem) {
    extern __shared__ __align__(16) unsigned char smG[];
    const int nq = d * D::BYTES / 16;                       // 16-byte vectors per row
    const int rows = 2 * H;
    const uint4* Wg_a = static_cast<const uint4*>(W_a);
    const uint4* Wg_b = static_cast<const uint4*>(W_b);
    uint4* Ws = reinterpret_cast<uint4*>(smG);              // [2H][nq]: W_a rows, then W_b rows
    if (use_smem) {
        for (int i = threadIdx.x; i < rows * nq; i += GG_THREADS) {
            const int r = i / nq, q = i - r * nq;
            Ws[i] = r < H ? __ldg(Wg_a + static_cast<int64_t>(r) * nq + q) : __ldg(Wg_b + static_cast<int64_t>(r - H) * nq + q);
        }
        __syncthreads();
    }
    const int lane = threadIdx.x & 31;
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (GG_THREADS / 32);
    for (int64_t u = static_cast<int64_t>(blockIdx.x) * (GG_THREADS / 32) + (threadIdx.x >> 5); u < tokens; u += wstride) {
        const uint4* xr = static_cast<const uint4*>(x) + u * nq;
        float acc[NH];
#pragma unroll
        for (int r = 0; r < NH; ++r) acc[r] = 0.f;
        for (int q = lane; q < nq; q += 32) {
            float fx[D::E];
            unpack16<D>(__ldg(xr + q), fx);
#pragma unroll
            for (int r = 0; r < NH; ++r) {
                if (r < rows) {
                    const uint4 wv = use_smem ? Ws[r * nq + q]
                                              : (r < H ? __ldg(Wg_a + static_cast<int64_t>(r) * nq + q)
                                                       : __ldg(Wg_b + static_cast<int64_t>(r - H) * nq + q));
                    float fw[D::E];
                    unpack16<D>(wv, fw);
#pragma unroll
                    for (int e = 0; e < D::E; ++e) acc[r] = fmaf(fw[e], fx[e], acc[r]);
                }
            }
        }
#pragma unroll
        for (int r = 0; r < NH; ++r) {
            if (r < rows) {
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], off);
            }
        }
        const int64_t b = u / T, t = u - b * T;
        for (int j = lane; j < rows; j += 32) {
            float z = 0.f;
#pragma unroll
            for (int r = 0; r < NH; ++r) z = (r == j) ? acc[r] : z;
            if (j < H) {
                const float za = z + __ldg(b_dt + j);
                const float sp = za > 20.f ? za : log1pf(expf(za));     // softplus
                store_elem<D>(alpha, (b * H + j) * T + t, expf(-__ldg(A + j) * sp));
            } else {
                store_elem<D>(beta, (b * H + (j - H)) * T + t, 1.f / (1.f + expf(-z)));
            }
        }
    }
}

// MC: 8-byte chunks per lane (row bytes <= 256 * MC).
template <class D, int MC>
__global__ void __launch_bounds__(GT_THREADS) k_norm_gate(const void* __restrict__ y, const void* __restrict__ g,
                                                          const float* __restrict__ gamma, float eps, void* __restrict__ z,
                                                          int64_t rows, int H, int T, int dv) {
    using C = Chunk8<D>;
    const int lane = threadIdx.x & 31;
    const int nc = dv / C::E;                               // 8-byte chunks per row
    const int64_t wstride = static_cast<int64_t>(gridDim.x) * (GT_THREADS / 32);
    for (int64_t u = static_cast<int64_t>(blockIdx.x) * (GT_THREADS / 32) + (threadIdx.x >> 5); u < rows; u += wstride) {
        const uint2* yr = static_cast<const uint2*>(y) + u * nc;
        const uint2* gr = static_cast<const uint2*>(g) + u * nc;
        float fy[MC][C::E];
        uint2 gv[MC];
        float ss = 0.f;
#pragma unroll
        for (int m = 0; m < MC; ++m) {                       // y and g of the row in flight together
            const int c = lane + 32 * m;
            if (c < nc) {
                gv[m] = __ldg(gr + c);
                C::unpack(__ldg(yr + c), fy[m]);
#pragma unroll
                for (int e = 0; e < C::E; ++e) ss = fmaf(fy[m][e], fy[m][e], ss);
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        const float inv = 1.f / sqrtf(ss / static_cast<float>(dv) + eps);
        // row u = (b * H + h) * T + t  ->  z row (b * T + t) * H + h
        const int64_t bh = u / T, t = u - bh * T;
        const int64_t b = bh / H, h = bh - b * H;
        uint2* zr = static_cast<uint2*>(z) + ((b * T + t) * H + h) * nc;
#pragma unroll
        for (int m = 0; m < MC; ++m) {
            const int c = lane + 32 * m;
            if (c < nc) {
                float fg[C::E], o[C::E];
                C::unpack(gv[m], fg);
#pragma unroll
                for (int e = 0; e < C::E; ++e) o[e] = fg[e] * __ldg(gamma + c * C::E + e) * (fy[m][e] * inv);
                zr[c] = C::pack(o);
            }
        }
    }
}

namespace {
unsigned persistent_grid(int64_t warps_wanted, int threads = GT_THREADS) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int64_t grid = (warps_wanted + threads / 32 - 1) / (threads / 32);
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * (2048 / threads);   // a full SM of threads
    return static_cast<unsigned>(grid < 1 ? 1 : (grid < cap ? grid : cap));
}

template <class D, int NH>
cudaError_t gates_nh(const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A, void* alpha,
                     void* beta, int B, int T, int H, int d, cudaStream_t s) {
    const size_t wbytes = static_cast<size_t>(2) * H * d * D::BYTES;
    const int use_smem = wbytes <= GT_SMEM_MAX;
    const size_t smem = use_smem ? wbytes : 0;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_gates<D, NH>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    const int64_t tokens = static_cast<int64_t>(B) * T;
    k_gates<D, NH><<<persistent_grid(tokens, GG_THREADS), GG_THREADS, smem, s>>>(x, W_a, W_b, b_dt, A, alpha, beta, tokens, T, H, d,
                                                                    use_smem);
    return cudaGetLastError();
}

template <class D>
cudaError_t gates_dtype(const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A, void* alpha,
                        void* beta, int B, int T, int H, int d, cudaStream_t s) {
    const int rows = 2 * H;
    if (rows <= 2) return gates_nh<D, 2>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, s);
    if (rows <= 8) return gates_nh<D, 8>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, s);
    if (rows <= 16) return gates_nh<D, 16>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, s);
    if (rows <= 32) return gates_nh<D, 32>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, s);
    return gates_nh<D, 64>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, s);
}

template <class D>
cudaError_t norm_gate_dtype(const void* y, const void* g, const float* gamma, float eps, void* z, int B, int H, int T,
                            int dv, cudaStream_t s) {
    const int nc = dv / Chunk8<D>::E;
    const int64_t rows = static_cast<int64_t>(B) * H * T;
    const unsigned grid = persistent_grid(rows);
    if (nc <= 32) k_norm_gate<D, 1><<<grid, GT_THREADS, 0, s>>>(y, g, gamma, eps, z, rows, H, T, dv);
    else if (nc <= 64) k_norm_gate<D, 2><<<grid, GT_THREADS, 0, s>>>(y, g, gamma, eps, z, rows, H, T, dv);
    else k_norm_gate<D, 4><<<grid, GT_THREADS, 0, s>>>(y, g, gamma, eps, z, rows, H, T, dv);
    return cudaGetLastError();
}
}  // namespace

cudaError_t launch_gates(int dtype, const void* x, const void* W_a, const void* W_b, const float* b_dt, const float* A,
                         void* alpha, void* beta, int B, int T, int H, int d, cudaStream_t stream) {
    return dtype == 0 ? gates_dtype<F32>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, stream)
                      : gates_dtype<BF16>(x, W_a, W_b, b_dt, A, alpha, beta, B, T, H, d, stream);
}

cudaError_t launch_norm_gate(int dtype, const void* y, const void* g, const float* gamma, float eps, void* z, int B, int H,
                             int T, int dv, cudaStream_t stream) {
    return dtype == 0 ? norm_gate_dtype<F32>(y, g, gamma, eps, z, B, H, T, dv, stream)
                      : norm_gate_dtype<BF16>(y, g, gamma, eps, z, B, H, T, dv, stream);
}

}  // namespace sdm
