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
// Persistent kernel, one CTA per SM, 512 threads (16 warps). Warp w owns TMEM
// lane quadrant w & 3 (pixels 32 (w & 3) .. + 31 of the tile) and quarter
// w >> 2 of the work on those pixels. Per tile:
//   TMA    z tile (c / 64 boxes of 64 x 128 bytes, 64-byte swizzle), two
//          buffers when shared memory allows, issued ahead of use;
//   limbs  each quarter writes both limbs of its quarter of K into TMEM
//          (the A operand, two fp16 per column);
//   MMA    c / 64 passes of 64 output channels, D_h and D_l by c / 16
//          K-steps each into accumulator buffer p & 1, so the MMAs of pass
//          p + 1 run while the threads finish pass p; G (the B operand) stays
//          in shared memory;
//   pool   each thread finishes 16 channels of its pixel per pass: the float
//          estimate of the code, exact 64-bit comparisons near a rounding
//          boundary, u into a shared-memory row;
//   out    after each pass, that pass's 64-channel group: four lanes per
//          pixel row, 16 values each, Sylvester block of u (int32, exact;
//          the two widest stages through lane shuffles), then a table of
//          clamp(round(M_in v / 2^n_in)) over |v| <= 127 hb built once per
//          CTA, 16-byte stores. The last group's transition runs next to the
//          next tile's limbs, whose MMAs then start early.
// Every wait is bounded; the CTA leaves its loop together after a failure.
#include <cuda_fp16.h>

#include "hatq_internal.h"
#include "hatq_tc.h"

namespace hatq {
namespace {

using namespace tc;

constexpr int kGdnThreads = 512;

// two values v0 (low half), v1 in [0, 1023] -> one fp16x2 word, exactly:
// 0x6400 | v is the fp16 pattern of 1024 + v
__device__ __forceinline__ uint32_t u10x2_to_f16x2(uint32_t v0, uint32_t v1) {
    const uint32_t t = (v0 | (v1 << 16)) | 0x64006400u;
    uint32_t r;
    asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x64006400u));
    return r;
}

__device__ __forceinline__ uint32_t prmt(uint32_t x, uint32_t y, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(x), "r"(y), "r"(sel));
    return d;
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}

// |u| for one channel, exactly: the largest k <= 127 with (2k - 1)^2 den <= num
// (GDN: den = D 2^t, num = 4 P a^2; IGDN: den = 2^t, num = 4 P a^2 D), i.e.
// round(X) with ties up for X = a sqrt(P / (2^t D)) (IGDN: a sqrt(P D / 2^t)),
// searched from the estimate k0 (the loops make it exact whatever k0 is).
__device__ __noinline__ int gdn_code_exact(uint32_t ab, uint32_t D, int k0, const GdnArgs &a) {
    unsigned long long num = 4ull * a.P * (unsigned long long)(ab * ab);
    unsigned long long den;
    if (a.inverse) {
        num *= D;
        den = 1ull << a.t;
    } else {
        den = (unsigned long long)D << a.t;
    }
    auto cond = [&](int kk) {
        const unsigned long long o = (unsigned long long)(2 * kk - 1);
        return o * o * den <= num;
    };
    int k = k0 < 0 ? 0 : (k0 > 127 ? 127 : k0);
    while (k < 127 && cond(k + 1)) ++k;
    while (k > 0 && !cond(k)) --k;
    return k;
}

// The code u of one channel from its pool (fp32 limb sums dh, dl of the
// tensor cores, exact integers) and its preactivation zi. The float estimate
// X = |z| sr rsqrt(D) (IGDN: |z| sr sqrt(D)), sr = sqrt(P / 2^t), has a
// relative error below 2^-21 (rsqrt within 2 ulp, five roundings of 2^-24),
// so below 2^-14 for X < 128: it decides every code whose X lies more than
// 2^-10 from a half-integer and below 126.5; the rest take the exact path.
__device__ __forceinline__ int gdn_code(int zi, float dh, float dl, float bf, const int32_t *bi, const GdnArgs &a) {
    const float zf = __int_as_float(0x4B000000 | (uint32_t)(zi + 128)) - 8388736.0f;   // exact
    const float df = fmaf(128.0f, dh, dl + bf);
    const float r = rsqrtf(df);
    const float x = a.inverse ? zf * a.sr * (df * r) : zf * a.sr * r;                   // signed X
    const float t = x + 12582912.0f;
    const float kf = t - 12582912.0f;
    if (fabsf(x - kf) < 0.4990234375f && fabsf(x) < 126.5f) return __float_as_int(t) - 0x4B400000;
    const uint32_t D = (__float2uint_rz(dh) << 7) + __float2uint_rz(dl) + (uint32_t)*bi;
    const int k = gdn_code_exact((uint32_t)abs(zi), D, (int)(fabsf(x) + 0.5f), a);
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
    const uint32_t gbar = bar0 + 16u;
    auto mma_bar = [&](int b) { return bar0 + 24u + 8u * b; };
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_area + 40);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_area + 44);
    const int ustride = c + 16;

    __shared__ int s_skip;
    if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int *>(a.err);
    __syncthreads();
    if (s_skip != 0) return;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quad = warp & 3, part = warp >> 2;            // lane quadrant, quarter of the work
    const int m = quad * 32 + lane;                         // pixel row of the tile
    const int my_tiles = a.num_tiles > (int)blockIdx.x ? (a.num_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

    if (threadIdx.x == 0) {
        mbar_init(zfull(0), 1);
        mbar_init(zfull(1), 1);
        mbar_init(gbar, 1);
        mbar_init(mma_bar(0), 1);
        mbar_init(mma_bar(1), 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_holder)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    float *bf_s = reinterpret_cast<float *>(b_s + c);
    for (int i = threadIdx.x; i < c; i += kGdnThreads) {
        b_s[i] = a.b_pool[i];
        bf_s[i] = (float)a.b_pool[i];
    }
    // x = clamp(round(M_in v / 2^n_in)) for every v = H~ u, |v| <= 127 hb; lut_s[v]
    const int vmax = 127 * (a.hb_next > 1 ? a.hb_next : 1);
    const int8_t *lut_s = reinterpret_cast<const int8_t *>(smem + a.lut_off) + vmax;
    for (int v = -vmax + (int)threadIdx.x; v <= vmax; v += kGdnThreads)
        const_cast<int8_t *>(lut_s)[v] = (int8_t)requant8_any(a.mult_in * (long long)v, a.shift_in);
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

    // TMEM: A limbs h, l at columns [0, c / 2), [c / 2, c); accumulator buffer
    // b at c + 128 b holds D_h (64 columns) and D_l (64 columns) of one pass,
    // i.e. 64 output channels; pass p uses buffer p & 1, so the MMAs of pass
    // p + 1 run while the threads finish pass p.
    const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16);
    const uint32_t idesc = idesc_f16(64);
    const uint64_t gdesc0 = sdesc_sw128(smem_addr(g_s));
    const int np = c / 64;
    bool ok = true;
    int issued = a.nz < my_tiles ? a.nz : my_tiles;
    uint32_t mph0 = 0, mph1 = 0;            // next phase parity of each accumulator barrier
    bool pend0 = false, pend1 = false;      // thread 0: a commit not yet waited for
    bool g_ready = false;
    // thread 0: the MMAs of pass p into buffer p & 1 and their commit
    auto issue_pass = [&](int p) {
        tc_fence_after();
        if (!g_ready) {
            g_ready = mbar_wait(gbar, 0, abort_flag, a.err);
            if (!g_ready) return;
        }
        const int b = p & 1;
        for (int limb = 0; limb < 2; ++limb) {
            const uint32_t d = tmem + (uint32_t)(c + 128 * b + 64 * limb);
            for (int s = 0; s < c / 16; ++s) {
                const uint64_t bd = gdesc0 + (uint64_t)(((uint32_t)p * 64u * 128u) >> 4) +
                                    (uint64_t)(((uint32_t)(s >> 2) * c * 128u) >> 4) + (uint64_t)(2 * (s & 3));
                umma_f16_ts(d, tmem + (uint32_t)(limb * (c / 2) + 8 * s), bd, idesc, s > 0 ? 1u : 0u);
            }
        }
        umma_commit(mma_bar(b));
        if (b) pend1 = true;
        else pend0 = true;
    };
    // ---- limbs of z^2 of this pixel row into TMEM: this quarter's K range, both limbs
    auto limbs = [&](const uint8_t *zt) {
        const int sw = (m >> 1) & 3;
        for (int k = part * (c / 4); k < (part + 1) * (c / 4); k += 16) {
            const uint4 v = *reinterpret_cast<const uint4 *>(zt + (k >> 6) * 8192 + m * 64 +
                                                              ((((k & 63) >> 4) ^ sw) << 4));
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
            uint32_t hh[8], ll[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int z0 = (int)(int8_t)(w[i >> 1] >> (16 * (i & 1)));
                const int z1 = (int)(int8_t)(w[i >> 1] >> (16 * (i & 1) + 8));
                const uint32_t s0 = (uint32_t)(z0 * z0), s1 = (uint32_t)(z1 * z1);
                hh[i] = u10x2_to_f16x2(s0 >> 7, s1 >> 7);
                ll[i] = u10x2_to_f16x2(s0 & 127u, s1 & 127u);
            }
            tmem_st8(t_lane + (uint32_t)(k / 2), hh);
            tmem_st8(t_lane + (uint32_t)(c / 2 + k / 2), ll);
        }
        tmem_wait_st();
    };
    // ---- pool and codes u of channels 64 p + 16 part .. + 15 of this pixel (accumulator buffer db)
    auto pool = [&](const uint8_t *zt, int p, int db) {
        const int sw = (m >> 1) & 3;
        const int col = 16 * part;                       // column within the pass
        const int ch = 64 * p + col;
        uint32_t dh[16], dl[16];
        tmem_ld16(t_lane + (uint32_t)(c + 128 * db + col), dh);
        tmem_ld16(t_lane + (uint32_t)(c + 128 * db + 64 + col), dl);
        const uint4 zv = *reinterpret_cast<const uint4 *>(zt + (ch >> 6) * 8192 + m * 64 +
                                                           ((((ch & 63) >> 4) ^ sw) << 4));
        float bfv[16];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 f4 = reinterpret_cast<const float4 *>(bf_s + ch)[q];
            bfv[4 * q] = f4.x; bfv[4 * q + 1] = f4.y; bfv[4 * q + 2] = f4.z; bfv[4 * q + 3] = f4.w;
        }
        tmem_wait_ld();
        const uint32_t zw[4] = {zv.x, zv.y, zv.z, zv.w};
        uint32_t out[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int u[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int e = 4 * q + i;
                const int zi = (int)(int8_t)(zw[q] >> (8 * i));
                u[i] = gdn_code(zi, __uint_as_float(dh[e]), __uint_as_float(dl[e]), bfv[e], b_s + ch + e, a);
            }
            out[q] = prmt(prmt((uint32_t)u[0], (uint32_t)u[1], 0x0040u), prmt((uint32_t)u[2], (uint32_t)u[3], 0x0040u),
                          0x5410u);
        }
        *reinterpret_cast<uint4 *>(u_s + m * ustride + ch) = make_uint4(out[0], out[1], out[2], out[3]);
    };
    // ---- input transition of the next layer on channel group p (64 channels) of
    // tile jt: four consecutive lanes share a pixel row, 16 values each; block
    // stages 1..8 in the lane, 16 and 32 across the four lanes; Sylvester block in
    // int32 (exact: |H~ u| <= 127 hb), then the table of clamp(round(M_in v / 2^n_in))
    auto transition = [&](int jt, int p) {
        const int r = (int)threadIdx.x >> 2, sub = (int)threadIdx.x & 3;
        const uint4 w = *reinterpret_cast<const uint4 *>(u_s + r * ustride + 64 * p + 16 * sub);
        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
        int v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = (int)(int8_t)(ww[i >> 2] >> (8 * (i & 3)));
        const int hb = a.hb_next;
        fwht<16>(v, hb < 16 ? hb : 16);
        for (int mm = 1; mm <= 2; mm <<= 1) {
            if (16 * mm >= hb) break;
            const bool upper = (sub & mm) != 0;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int q = __shfl_xor_sync(0xffffffffu, v[i], mm);
                v[i] = upper ? q - v[i] : v[i] + q;
            }
        }
        const long long pix = (long long)((int)blockIdx.x + jt * (int)gridDim.x) * 128 + r;
        if (pix < a.pixels) {
            uint32_t wd[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
                wd[q] = prmt(prmt((uint32_t)lut_s[v[4 * q]], (uint32_t)lut_s[v[4 * q + 1]], 0x0040u),
                             prmt((uint32_t)lut_s[v[4 * q + 2]], (uint32_t)lut_s[v[4 * q + 3]], 0x0040u), 0x5410u);
            *reinterpret_cast<uint4 *>(a.y + pix * c + 64 * p + 16 * sub) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        }
    };

    // Schedule per tile: [MMA wait, pool of pass p, barrier, MMAs of pass p + 2,
    // transition of group p] for each pass, except that the last group's
    // transition runs next to the limbs of the next tile, whose first MMAs then
    // start while this tile's last writes drain.
    int j = 0;
    if (my_tiles > 0) {
        ok = __syncthreads_and(mbar_wait(zfull(0), 0, abort_flag, a.err));
        if (ok) {
            limbs(z_s);
            tc_fence_before();
            __syncthreads();
            if (threadIdx.x == 0) {
                issue_pass(0);
                if (np > 1) issue_pass(1);
            }
        }
    }
    for (; j < my_tiles && ok; ++j) {
        const uint8_t *zt = z_s + (size_t)(j % a.nz) * zbytes;
        for (int p = 0; p < np && ok; ++p) {
            const int db = p & 1;
            ok = __syncthreads_and(mbar_wait(mma_bar(db), db ? mph1 : mph0, abort_flag, a.err));
            if (db) { mph1 ^= 1u; pend1 = false; }
            else { mph0 ^= 1u; pend0 = false; }
            if (!ok) break;
            tc_fence_after();
            pool(zt, p, db);
            tc_fence_before();
            __syncthreads();                               // codes of group p complete; buffer db free
            if (threadIdx.x == 0 && p + 2 < np) issue_pass(p + 2);
            if (p + 1 < np) transition(j, p);
        }
        if (!ok) break;
        // every pool of this tile is done: its z buffer takes the tile that reuses it
        if (threadIdx.x == 0 && issued < my_tiles) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_z(issued);
            ++issued;
        }
        transition(j, np - 1);
        if (j + 1 < my_tiles) {
            const int b1 = (j + 1) % a.nz;
            ok = __syncthreads_and(mbar_wait(zfull(b1), (uint32_t)(((j + 1) / a.nz) & 1), abort_flag, a.err));
            if (!ok) break;
            limbs(z_s + (size_t)b1 * zbytes);              // the A columns are free: pass np - 1 was waited for
            tc_fence_before();
            __syncthreads();
            if (threadIdx.x == 0) {
                issue_pass(0);
                if (np > 1) issue_pass(1);
            }
        }
    }
    // after a failure: wait (bounded) for this CTA's copies and MMAs in flight
    if (!ok && threadIdx.x == 0) {
        const long long t0 = clock64();
        if (pend0)
            while (!mbar_try_wait(mma_bar(0), mph0) && clock64() - t0 < kWaitLimitCycles) {
            }
        if (pend1)
            while (!mbar_try_wait(mma_bar(1), mph1) && clock64() - t0 < kWaitLimitCycles) {
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
