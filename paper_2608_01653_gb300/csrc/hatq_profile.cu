// Profiling pass of HaTQ's layer-wise strategy selection (Eq.
// hadamard_sensitivity): for each image of an NHWC INT8 code tensor, max|x|
// and max|H~_hb x| over the whole image, in one read of the tensor.
//
// Memory-bound. A warp owns a 512-element span of one image (16 codes per
// lane, one 16-byte load), so every Hadamard block (hb | C, 16 | C) lies in
// one warp. Codes and every partial sum of the Sylvester butterfly are
// integers of magnitude <= 127 * 256 < 2^24, so the butterfly runs exactly in
// fp32 on the FMA pipe: a code b becomes fp32 through the mantissa
// (bits 0x4B000000 | (b + 128) are 2^23 + b + 128), in-lane stages are
// adds/subtracts and cross-lane stages a shuffle and a multiply-add by +-1.
// The indicator max|H~ x|^2 > hb max|x|^2 (||T x||_inf > ||x||_inf for the
// normalized transform) is then decided exactly in 64-bit integers.
#include "hatq_internal.h"

namespace hatq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// 16 codes -> 16 exact fp32 values.
__device__ __forceinline__ void decode16(const int4 raw, float (&v)[16]) {
    const uint32_t w[4] = {(uint32_t)raw.x, (uint32_t)raw.y, (uint32_t)raw.z, (uint32_t)raw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t u = w[i] ^ 0x80808080u;   // b + 128 in every byte
#pragma unroll
        for (int k = 0; k < 4; ++k)
            v[4 * i + k] = __uint_as_float(prmt(u, 0x4B000000u, 0x7650u + (uint32_t)k)) - 8388736.0f;   // - (2^23 + 128)
    }
}

__device__ __forceinline__ void butterfly(float (&v)[16], int hb, int lane) {
#pragma unroll
    for (int h = 1; h < 16; h <<= 1) {
        if (h >= hb) break;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            if (i & h) continue;
            const float a = v[i], b = v[i + h];
            v[i] = a + b;
            v[i + h] = a - b;
        }
    }
#pragma unroll
    for (int m = 1; m < 16; m <<= 1) {
        if (16 * m >= hb) break;
        const float sgn = (lane & m) ? -1.0f : 1.0f;   // upper lane of a pair keeps partner - own
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float p = __shfl_xor_sync(0xffffffffu, v[i], m);
            v[i] = fmaf(sgn, v[i], p);
        }
    }
}

__global__ void __launch_bounds__(kThreads) profile_kernel(ProfileArgs a) {
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    const long long E = a.per_image;
    const long long tiles = (E + 511) >> 9;
    const long long first = (long long)blockIdx.x * (kThreads / 32) + wib;
    const long long stride = (long long)gridDim.x * (kThreads / 32);
    for (int img = blockIdx.y; img < a.n; img += gridDim.y) {
        const int8_t *xi = a.x + (long long)img * E;
        auto load = [&](long long t) {
            const long long e0 = (t << 9) + lane * 16;
            return (t < tiles && e0 < E) ? __ldg(reinterpret_cast<const int4 *>(xi + e0)) : make_int4(0, 0, 0, 0);
        };
        float mx = 0.f, mh = 0.f;
        int4 cur = load(first);
        for (long long t = first; t < tiles; t += stride) {
            const int4 nxt = load(t + stride);        // next tile in flight during this one
            float v[16];
            decode16(cur, v);
#pragma unroll
            for (int i = 0; i < 16; ++i) mx = fmaxf(mx, fabsf(v[i]));
            butterfly(v, a.hb, lane);
#pragma unroll
            for (int i = 0; i < 16; ++i) mh = fmaxf(mh, fabsf(v[i]));
            cur = nxt;
        }
        const int imx = __reduce_max_sync(0xffffffffu, (int)mx);
        const int imh = __reduce_max_sync(0xffffffffu, (int)mh);
        if (lane == 0) {
            if (imx) atomicMax(&a.maxima[2 * img], imx);
            if (imh) atomicMax(&a.maxima[2 * img + 1], imh);
        }
    }
}

__global__ void profile_finalize_kernel(const int *maxima, uint8_t *expands, int n, int hb) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const long long m = maxima[2 * i], h = maxima[2 * i + 1];
    expands[i] = (uint8_t)(h * h > (long long)hb * m * m);
}

}  // namespace

cudaError_t launch_profile(const ProfileArgs &a, uint8_t *expands, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(a.maxima, 0, sizeof(int) * 2 * (size_t)a.n, s);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
    const long long tiles = (a.per_image + 511) / 512;
    const int gy = a.n < 65535 ? a.n : 65535;
    const long long want = ((long long)sms * 8 + gy - 1) / gy;          // about 8 resident blocks per SM overall
    const long long need = (tiles + (kThreads / 32) - 1) / (kThreads / 32);
    const int gx = (int)(want < need ? (want < 1 ? 1 : want) : (need < 1 ? 1 : need));
    profile_kernel<<<dim3(gx, gy), kThreads, 0, s>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (expands) {
        profile_finalize_kernel<<<(a.n + 255) / 256, 256, 0, s>>>(a.maxima, expands, a.n, a.hb);
        e = cudaGetLastError();
    }
    return e;
}

}  // namespace hatq
