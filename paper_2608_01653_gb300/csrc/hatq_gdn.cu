// The GDN / IGDN transition of the supplementary's general nonlinearities
// (Eqs. supp_general_activation, supp_general_input_scale,
// supp_general_input_transition) for channel-coupled activations, on the
// 5th-generation tensor cores.
//
// Input: the integer preactivation z (Eq. supp_general_preactivation), one
// row of c INT8 codes per pixel, as a plain layer with output scale s_z emits
// it. Per pixel:
//   D_i = B_i + sum_j G_ij z_j^2                        (the normalization pool)
//   |u_i| = largest k <= 127 with (2k - 1)^2 D_i 2^t <= 4 P z_i^2     (GDN)
//           largest k <= 127 with (2k - 1)^2 2^t <= 4 P z_i^2 D_i     (IGDN)
//   u_i with the sign of z_i, i.e. round(R |z_i| / sqrt(D_i)) (IGDN: times
//   sqrt(D_i)) with ties away from zero and R^2 = P / 2^t;
//   x = clamp(round(H~_next (M_in u) / 2^n_in), -127, 127).
//
// The pool is a dense contraction over channels: D = Z2 G^T for a tile of
// 128 pixels, Z2 the squared codes. z^2 <= 16129 is split into two limbs
// h = z^2 >> 7 and l = z^2 & 127, both exact in fp16, and G <= 511 is exact in
// fp16; every product is <= 511 * 127 and a sum over c <= 256 channels stays
// below 2^24, so the two fp32 accumulators D_h, D_l in tensor memory hold
// exact integers and D = 128 D_h + D_l + B.
//
// Persistent kernel, 256 threads (8 warps). Warp w owns TMEM lane quadrant
// w & 3 (pixels 32 (w & 3) .. + 31 of the tile) and half w >> 2 of the work
// on those pixels. Per tile:
//   TMA    z tile (c / 64 boxes of 64 x 128 bytes, 64-byte swizzle), two
//          buffers when shared memory allows, issued one tile ahead;
//   limbs  half 0 writes limb h, half 1 limb l into TMEM (A operand);
//   MMA    for each half of the output channels (N = c / 2): D_h, D_l by
//          c / 16 K-steps each, G (B operand) resident in shared memory;
//   pool   each thread finishes c / 4 channels of its pixel: D, then u
//          (float estimate of k, corrected by exact 64-bit comparisons),
//          into a shared-memory row;
//   out    64-channel groups of u: Sylvester transform (int32, exact),
//          M_in multiply and one round-shift, 16-byte stores.
// Every wait is bounded; the CTA leaves its loop together after a failure.
#include <cuda_fp16.h>

#include "hatq_internal.h"
#include "hatq_tc.h"

namespace hatq {
namespace {

using namespace tc;

constexpr int kGdnThreads = 256;

// two values v0 (low half), v1 in [0, 1023] -> one fp16x2 word, exactly:
// 0x6400 | v is the fp16 pattern of 1024 + v
__device__ __forceinline__ uint32_t u10x2_to_f16x2(uint32_t v0, uint32_t v1) {
    const uint32_t t = (v0 | (v1 << 16)) | 0x64006400u;
    uint32_t r;
    asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x64006400u));
    return r;
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// an fp32 accumulator holding an exact integer in [0, 2^24) -> its value
__device__ __forceinline__ uint32_t acc_int(uint32_t bits) { return __float2uint_rz(__uint_as_float(bits)); }

// |u| for one channel: the largest k <= 127 with (2k - 1)^2 den <= num
// (GDN: den = D 2^t, num = 4 P a^2; IGDN: den = 2^t, num = 4 P a^2 D).
// The float estimate is exact to well under one code; the loops make the
// result exact whatever the estimate.
__device__ __forceinline__ int gdn_code(int zi, uint32_t D, const GdnArgs &a) {
    if (zi == 0) return 0;
    const uint32_t ab = (uint32_t)abs(zi);
    unsigned long long num = 4ull * a.P * (unsigned long long)(ab * ab);
    unsigned long long den;
    float x;
    if (a.inverse) {
        num *= D;
        den = 1ull << a.t;
        x = (float)ab * sqrtf(a.r2f * (float)D);
    } else {
        den = (unsigned long long)D << a.t;
        x = (float)ab * sqrtf(a.r2f / (float)D);
    }
    int k = (int)fminf(x + 0.5f, 127.f);
    auto cond = [&](int kk) {
        const unsigned long long o = (unsigned long long)(2 * kk - 1);
        return o * o * den <= num;
    };
    while (k < 127 && cond(k + 1)) ++k;
    while (k > 0 && !cond(k)) --k;
    return zi < 0 ? -k : k;
}

__global__ void __launch_bounds__(kGdnThreads, 1)
    gdn_kernel(const __grid_constant__ CUtensorMap tmZ, const __grid_constant__ CUtensorMap tmG,
               const __grid_constant__ GdnArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int c = a.c;
    const int zbytes = 128 * c;
    uint8_t *g_s = smem;                                   // [c / 64][c rows][128 B], 128-byte swizzle
    uint8_t *z_s = smem + a.z_off;                         // nz x [c / 64][128 rows][64 B], 64-byte swizzle
    uint8_t *u_s = smem + a.u_off;                         // [128 rows][c + 16 B]
    int32_t *b_s = reinterpret_cast<int32_t *>(smem + a.b_off);
    uint8_t *bar_area = smem + a.bar_off;
    const uint32_t bar0 = smem_addr(bar_area);
    auto zfull = [&](int b) { return bar0 + 8u * b; };
    const uint32_t gbar = bar0 + 16u, mma_bar = bar0 + 24u;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_area + 32);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_area + 36);
    const int ustride = c + 16;

    __shared__ int s_skip;
    if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int *>(a.err);
    __syncthreads();
    if (s_skip != 0) return;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quad = warp & 3, half = warp >> 2;
    const int m = quad * 32 + lane;                         // pixel row of the tile
    const int my_tiles = a.num_tiles > (int)blockIdx.x ? (a.num_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

    if (threadIdx.x == 0) {
        mbar_init(zfull(0), 1);
        mbar_init(zfull(1), 1);
        mbar_init(gbar, 1);
        mbar_init(mma_bar, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_holder)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    for (int i = threadIdx.x; i < c; i += kGdnThreads) b_s[i] = a.b_pool[i];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;

    auto issue_z = [&](int j) {
        const int b = j % a.nz;
        const int tile = (int)blockIdx.x + j * (int)gridDim.x;
        mbar_expect_tx(zfull(b), (uint32_t)zbytes);
        for (int cb = 0; cb < c / 64; ++cb)
            tma_load_2d(smem_addr(z_s + (size_t)b * zbytes + cb * 8192), &tmZ, zfull(b), 64 * cb, 128 * tile);
    };
    if (threadIdx.x == 0 && my_tiles > 0) {
        mbar_expect_tx(gbar, (uint32_t)(c * c * 2));
        for (int kb = 0; kb < c / 64; ++kb) tma_load_2d(smem_addr(g_s + kb * c * 128), &tmG, gbar, 64 * kb, 0);
        for (int j = 0; j < a.nz && j < my_tiles; ++j) issue_z(j);
    }

    // TMEM: A limbs h, l at columns [0, c / 2), [c / 2, c); D_h, D_l at [c, 3c / 2), [3c / 2, 2c)
    const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16);
    const uint32_t idesc = idesc_f16(c / 2);
    const uint64_t gdesc0 = sdesc_sw128(smem_addr(g_s));
    bool ok = true;
    int issued = a.nz < my_tiles ? a.nz : my_tiles;
    uint32_t mma_ph = 0;
    int j = 0;
    for (; j < my_tiles && ok; ++j) {
        const int b = j % a.nz;
        const uint8_t *zt = z_s + (size_t)b * zbytes;
        ok = __syncthreads_and(mbar_wait(zfull(b), (uint32_t)((j / a.nz) & 1), abort_flag, a.err));
        if (!ok) break;
        // ---- limbs of z^2 for this pixel row into TMEM
        {
            const int sw = (m >> 1) & 3;
            for (int k0 = 0; k0 < c; k0 += 32) {
                uint32_t cols[16];
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const int k = k0 + 16 * q;
                    const uint4 v = *reinterpret_cast<const uint4 *>(zt + (k >> 6) * 8192 + m * 64 +
                                                                      ((((k & 63) >> 4) ^ sw) << 4));
                    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int z0 = (int)(int8_t)(w[i >> 1] >> (16 * (i & 1)));
                        const int z1 = (int)(int8_t)(w[i >> 1] >> (16 * (i & 1) + 8));
                        const uint32_t s0 = (uint32_t)(z0 * z0), s1 = (uint32_t)(z1 * z1);
                        cols[8 * q + i] = half == 0 ? u10x2_to_f16x2(s0 >> 7, s1 >> 7)
                                                    : u10x2_to_f16x2(s0 & 127u, s1 & 127u);
                    }
                }
                tmem_st16(t_lane + (uint32_t)(half * (c / 2) + k0 / 2), cols);
            }
            tmem_wait_st();
        }
        tc_fence_before();
        __syncthreads();
        for (int nh = 0; nh < 2 && ok; ++nh) {
            // ---- MMA: D_h, D_l for output channels [nh c / 2, (nh + 1) c / 2)
            if (threadIdx.x == 0) {
                tc_fence_after();
                bool gok = true;
                if (j == 0 && nh == 0) gok = mbar_wait(gbar, 0, abort_flag, a.err);
                if (gok) {
                    for (int limb = 0; limb < 2; ++limb) {
                        const uint32_t d = tmem + (uint32_t)(c + limb * (c / 2));
                        for (int s = 0; s < c / 16; ++s) {
                            const uint64_t bd = gdesc0 + (uint64_t)(((uint32_t)nh * (c / 2) * 128u) >> 4) +
                                                (uint64_t)(((uint32_t)(s >> 2) * c * 128u) >> 4) + (uint64_t)(2 * (s & 3));
                            umma_f16_ts(d, tmem + (uint32_t)(limb * (c / 2) + 8 * s), bd, idesc, s > 0 ? 1u : 0u);
                        }
                    }
                    umma_commit(mma_bar);
                }
            }
            ok = __syncthreads_and(mbar_wait(mma_bar, mma_ph, abort_flag, a.err));
            mma_ph ^= 1u;
            if (!ok) break;
            tc_fence_after();
            // ---- pool and codes u for this thread's c / 4 channels of the half
            const int ch0 = nh * (c / 2) + half * (c / 4);
            const int sw = (m >> 1) & 3;
            for (int g0 = 0; g0 < c / 4; g0 += 16) {
                const int ch = ch0 + g0;
                uint32_t dh[16], dl[16];
                tmem_ld16(t_lane + (uint32_t)(c + (ch - nh * (c / 2))), dh);
                tmem_ld16(t_lane + (uint32_t)(c + c / 2 + (ch - nh * (c / 2))), dl);
                tmem_wait_ld();
                const uint4 zv = *reinterpret_cast<const uint4 *>(zt + (ch >> 6) * 8192 + m * 64 +
                                                                   ((((ch & 63) >> 4) ^ sw) << 4));
                const uint32_t zw[4] = {zv.x, zv.y, zv.z, zv.w};
                uint32_t out[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t word = 0;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int e = 4 * q + i;
                        const int zi = (int)(int8_t)(zw[q] >> (8 * i));
                        const uint32_t D = (acc_int(dh[e]) << 7) + acc_int(dl[e]) + (uint32_t)b_s[ch + e];
                        word |= ((uint32_t)gdn_code(zi, D, a) & 0xFFu) << (8 * i);
                    }
                    out[q] = word;
                }
                *reinterpret_cast<uint4 *>(u_s + m * ustride + ch) = make_uint4(out[0], out[1], out[2], out[3]);
            }
            tc_fence_before();
            __syncthreads();
        }
        if (!ok) break;
        // the z buffer is free: prefetch the tile that reuses it
        if (threadIdx.x == 0 && issued < my_tiles) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_z(issued);
            ++issued;
        }
        // ---- input transition of the next layer, 64-channel groups
        const long long pix = (long long)((int)blockIdx.x + j * (int)gridDim.x) * 128 + m;
        for (int grp = half; grp < c / 64; grp += 2) {
            int v[64];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 w = *reinterpret_cast<const uint4 *>(u_s + m * ustride + 64 * grp + 16 * q);
                const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int i = 0; i < 16; ++i) v[16 * q + i] = (int)(int8_t)(ww[i >> 2] >> (8 * (i & 3)));
            }
            fwht<64>(v, a.hb_next);
            if (pix < a.pixels) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t wd[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int e = 16 * q + 4 * i;
                        wd[i] = pack4(requant8_any(a.mult_in * (long long)v[e], a.shift_in),
                                      requant8_any(a.mult_in * (long long)v[e + 1], a.shift_in),
                                      requant8_any(a.mult_in * (long long)v[e + 2], a.shift_in),
                                      requant8_any(a.mult_in * (long long)v[e + 3], a.shift_in));
                    }
                    *reinterpret_cast<uint4 *>(a.y + pix * c + 64 * grp + 16 * q) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
                }
            }
        }
        __syncthreads();                                   // u rows are rewritten by the next tile
    }
    // after a failure: wait (bounded) for this CTA's copies and MMAs in flight
    if (!ok && threadIdx.x == 0) {
        const long long t0 = clock64();
        while (!mbar_try_wait(mma_bar, mma_ph ^ 1u) && clock64() - t0 < kWaitLimitCycles) {
        }
        if (my_tiles > 0)
            while (!mbar_try_wait(gbar, 0) && clock64() - t0 < kWaitLimitCycles) {
            }
        for (int jj = j; jj < issued; ++jj)
            while (!mbar_try_wait(zfull(jj % a.nz), (uint32_t)((jj / a.nz) & 1)) && clock64() - t0 < kWaitLimitCycles) {
            }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(a.tmem_cols) : "memory");
    }
}

}  // namespace

// Grid: the resident CTAs of every SM (limited by registers, shared memory
// and the 512 tensor-memory columns), at most one per tile.
cudaError_t launch_gdn(const CUtensorMap &tmZ, const CUtensorMap &tmG, const GdnArgs &a, int smem_bytes, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(gdn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, occ = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, gdn_kernel, kGdnThreads, smem_bytes)) != cudaSuccess)
        return e;
    const int per_sm = max(1, min(occ, 512 / a.tmem_cols));
    const int grid = (int)min((long long)a.num_tiles, (long long)sms * per_sm);
    gdn_kernel<<<grid, kGdnThreads, smem_bytes, s>>>(tmZ, tmG, a);
    return cudaGetLastError();
}

}  // namespace hatq
