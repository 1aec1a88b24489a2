// Shared device-side helpers of the SDM kernels (storage dtypes, 16-byte row chunks).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <math.h>

namespace sdm {

// Storage dtype traits.  A memory row is moved as 16-byte chunks of E elements.
struct F32 {
    using T = float;
    static constexpr int E = 4;
    static constexpr int BYTES = 4;
};
struct BF16 {
    using T = __nv_bfloat16;
    static constexpr int E = 8;
    static constexpr int BYTES = 2;
};

template <class D> __device__ __forceinline__ void unpack16(const uint4& u, float* f);
template <> __device__ __forceinline__ void unpack16<F32>(const uint4& u, float* f) {
    f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
}
template <> __device__ __forceinline__ void unpack16<BF16>(const uint4& u, float* f) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        f[2 * q] = __uint_as_float(w[q] << 16);
        f[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
    }
}

// fp32 -> storage, round-to-nearest-even.
template <class D> __device__ __forceinline__ uint4 pack16(const float* f);
template <> __device__ __forceinline__ uint4 pack16<F32>(const float* f) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]), __float_as_uint(f[3]));
}
template <> __device__ __forceinline__ uint4 pack16<BF16>(const float* f) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * q], f[2 * q + 1]);
        w[q] = *reinterpret_cast<uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// The same, as fp32 pairs (element 2q in .x, 2q + 1 in .y) for the packed fp32x2 units.
template <class D> __device__ __forceinline__ void unpack16x2(const uint4& u, float2* f);
template <> __device__ __forceinline__ void unpack16x2<F32>(const uint4& u, float2* f) {
    f[0] = make_float2(__uint_as_float(u.x), __uint_as_float(u.y));
    f[1] = make_float2(__uint_as_float(u.z), __uint_as_float(u.w));
}
template <> __device__ __forceinline__ void unpack16x2<BF16>(const uint4& u, float2* f) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) f[q] = make_float2(__uint_as_float(w[q] << 16), __uint_as_float(w[q] & 0xffff0000u));
}
template <class D> __device__ __forceinline__ uint4 pack16x2(const float2* f);
template <> __device__ __forceinline__ uint4 pack16x2<F32>(const float2* f) {
    return make_uint4(__float_as_uint(f[0].x), __float_as_uint(f[0].y), __float_as_uint(f[1].x), __float_as_uint(f[1].y));
}
template <> __device__ __forceinline__ uint4 pack16x2<BF16>(const float2* f) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        __nv_bfloat162 h = __floats2bfloat162_rn(f[q].x, f[q].y);
        w[q] = *reinterpret_cast<uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// One storage element -> fp32 (exact).
template <class D> __device__ __forceinline__ float load_elem(const void* base, int64_t i);
template <> __device__ __forceinline__ float load_elem<F32>(const void* base, int64_t i) {
    return __ldg(reinterpret_cast<const float*>(base) + i);
}
template <> __device__ __forceinline__ float load_elem<BF16>(const void* base, int64_t i) {
    const unsigned short b = __ldg(reinterpret_cast<const unsigned short*>(base) + i);
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// Device status word bits (read and cleared by sdm_device_status).
enum : int { ERR_BAD_INDEX = 1, ERR_UNSORTED = 2, ERR_TIMEOUT = 4, ERR_SELECT = 8 };

__device__ __forceinline__ void flag_error(int* err, int bit) {
    if (err) atomicOr(err, bit);
}

// Event counters stored after the status word (read and cleared by sdm_device_stats).
enum : int {
    STAT_HALF_BAND = 1,      // a half's top-k boundary was not certified by the fp32 scores
    STAT_HALF_FULL = 2,      // ... and its band reached past the kept list (whole half rescanned)
    STAT_COMB_BAND = 3,      // the outer-sum boundary was not certified by the fp32 scores
    STAT_COMB_FULL = 4,      // ... and its band reached past 64 candidates (serial float64)
    STAT_SELECT_RETRY = 5,   // a warp's survivor buffer overflowed once (tensor-core path)
    STAT_COMB_MERGE = 6,     // the outer-sum band reached the L-th candidate: merge extended to 64
    STAT_BAND_F64 = 7,       // a band near-tie was decided by float64 rescoring
    STAT_SERIAL = 8,         // the serial float64 fallback ran (heavy ties)
    STAT_HALF_BAND_ENTRIES = 9,   // sum over half bands of the entries rescored
    STAT_COMB_BAND_ENTRIES = 10,  // sum over outer-sum bands of the entries rescored
    STAT_COUNT = 11
};
__device__ __forceinline__ void stat_add(int* err, int which, unsigned n = 1u) {
    if (err) atomicAdd(reinterpret_cast<unsigned*>(err) + which, n);
}

}  // namespace sdm
