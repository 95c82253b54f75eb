// INT8 implicit-GEMM convolution with the fused requantize / Hadamard
// epilogue of HaTQ (Eqs. linear_operator, integer_accumulation,
// integer_hadamard_transition), on the 5th-generation tensor cores.
//
// GEMM view: rows = output pixels (M), columns = output channels (N),
// reduction K = (kh, kw, c_in) in that order, i.e. NHWC im2col order.
//
// Exact integer arithmetic on sm_103a. The tcgen05 integer kind does not exist
// on sm_103a, so the INT8 codes (|q| <= 127) are carried as IEEE fp16 values,
// which represent them exactly, and multiplied by tcgen05.mma kind::f16 into
// fp32 accumulators in tensor memory (TMEM). Every product is an integer of
// magnitude <= 127^2 and every partial sum of a 1024-long reduction chunk is
// an integer of magnitude <= 1024 * 127^2 < 2^24, so all fp32 values involved
// are exactly representable integers and the chunk sum is exact. Chunk g
// accumulates in TMEM region g & 1; the epilogue warps convert finished chunks
// to int32 and add them into int32 partials in their registers, so the full
// accumulator is the exact int32 sum.
//
// Persistent kernel, one CTA per SM, 512 threads in four warpgroups:
//   warp 0      TMA producer: weight tile (fp16, 128B-swizzled) and, for
//               c_in % 16 == 0, the INT8 activation box of one kernel tap and
//               64 input channels (64B-swizzled; zero fill outside the image =
//               zero padding), SUB 64-wide blocks per pipeline stage.
//   warp 1      TMEM allocation; lane 0 issues the MMAs (A operand in TMEM,
//               B in shared memory) and commits.
//   warps 2-3   idle (they complete warpgroup 0 for the register split).
//   warps 4-11  epilogue warpgroups: drains and the fused requantize /
//               Hadamard epilogue into a shared-memory output tile, copied out
//               coalesced.
//   warps 12-15 converters, one per TMEM lane quadrant: INT8 row -> fp16 pairs
//               in a TMEM slot ring (for small c_in, gathered from the tile's
//               input window staged in shared memory).
// Every mbarrier wait is bounded: on expiry the kernel records an error word,
// raises a CTA-wide abort flag and unwinds (waiting, again bounded, for its own
// MMAs and copies) before freeing TMEM.
// This file is compiled twice: as itself (the kernels for activation blocks of
// whole 64-channel boxes, the launcher, the self test) and, through
// hatq_conv_pieces.cu with HATQ_CONV_PIECES = 1, for the kernels whose blocks
// arrive as two 32-channel boxes; two translation units build in parallel.
#ifndef HATQ_CONV_PIECES
#define HATQ_CONV_PIECES 0
#endif

#include <cuda_fp16.h>

#include "hatq_internal.h"
#include "hatq_tc.h"

namespace hatq {
namespace {

using namespace tc;

constexpr int kThreads = 512;
constexpr int kConvThreads = 128;      // converter warps 12-15, one per TMEM lane quadrant

// 4 int8 codes (one 32-bit word) -> 2 fp16x2 words, exactly: with u = b + 128
// in [0, 255], the fp16 bit pattern 0x6400 | u is 1024 + u, and subtracting
// 1152 leaves b (every step is exact in fp16).
__device__ __forceinline__ void i8x4_to_f16x4(uint32_t w, uint32_t &lo, uint32_t &hi) {
    uint32_t u = w ^ 0x80808080u, a, b;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(a) : "r"(u), "r"(0x64646464u), "r"(0x4140u));
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(b) : "r"(u), "r"(0x64646464u), "r"(0x4342u));
    asm("sub.f16x2 %0, %1, %2;" : "=r"(lo) : "r"(a), "r"(0x64806480u));
    asm("sub.f16x2 %0, %1, %2;" : "=r"(hi) : "r"(b), "r"(0x64806480u));
}

// two int16 codes c0 (low half) and c1 in [-255, 255] -> one fp16x2 word,
// exactly: offset binary c + 32768 minus 32512 gives c + 256 in [1, 511] per
// half (no borrow between halves), 0x6400 | (c + 256) is 1024 + 256 + c, and
// subtracting 1280 leaves c.
__device__ __forceinline__ uint32_t i16x2_to_f16x2(uint32_t w) {
    const uint32_t t = ((w ^ 0x80008000u) - 0x7F007F00u) | 0x64006400u;
    uint32_t r;
    asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x65006500u));
    return r;
}

struct EpiCtx {
    const int *b_int;    // this tile's bias codes, multipliers and dequant factors (shared memory)
    const int *mult;
    const float *deq;
    const float *biasf;  // float bias added after the scale (dynamic affine input), else zeros
    uint32_t t_acc;      // TMEM address of this warp's lanes, column 0 of the accumulator
    bool int_acc;        // the accumulator holds exact int32 totals (else exact fp32 integers)
    uint8_t *row;        // this thread's row of the shared-memory output tile (INT8 output)
    float *gout;         // float32 output: this thread's pixel row in global memory, or null
    const int8_t *lut;   // general transition: phi_int table (shared memory), index z + 127
};

// Exact int32 accumulator of 16 columns starting at tile column `col`, bias included.
__device__ __forceinline__ void load_acc16(const EpiCtx &e, int col, int (&v)[16]) {
    uint32_t r[16];
    tmem_ld16(e.t_acc + col, r);
    tmem_wait_ld();
    if (e.int_acc) {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = (int)r[i];
    } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = __float2int_rn(__uint_as_float(r[i]));
    }
    const int4 *bp = reinterpret_cast<const int4 *>(e.b_int + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int4 b = bp[i];
        v[4 * i] += b.x; v[4 * i + 1] += b.y; v[4 * i + 2] += b.z; v[4 * i + 3] += b.w;
    }
}

// t = M (.) a for 16 columns starting at tile column col.
__device__ __forceinline__ void scale_i64(const EpiCtx &e, int col, const int (&v)[16], long long *t) {
    const int4 *mp = reinterpret_cast<const int4 *>(e.mult + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int4 m = mp[i];
        t[4 * i] = (long long)m.x * v[4 * i];
        t[4 * i + 1] = (long long)m.y * v[4 * i + 1];
        t[4 * i + 2] = (long long)m.z * v[4 * i + 2];
        t[4 * i + 3] = (long long)m.w * v[4 * i + 3];
    }
}
__device__ __forceinline__ void scale_f32(const EpiCtx &e, int col, const int (&v)[16], float *t) {
    const float4 *dp = reinterpret_cast<const float4 *>(e.deq + col);
    const float4 *bp = reinterpret_cast<const float4 *>(e.biasf + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float4 d = dp[i], b = bp[i];
        t[4 * i] = d.x * (float)v[4 * i] + b.x;
        t[4 * i + 1] = d.y * (float)v[4 * i + 1] + b.y;
        t[4 * i + 2] = d.z * (float)v[4 * i + 2] + b.z;
        t[4 * i + 3] = d.w * (float)v[4 * i + 3] + b.w;
    }
}

// Requantized codes of G columns starting at tile column col, written to this
// thread's row of the shared-memory output tile (copied out coalesced later).
template <int G>
__device__ __forceinline__ void store_codes(const ConvArgs &a, uint8_t *row, int col, const long long (&t)[G]) {
    if (a.shift >= 32) {
        // lower clamp in the round-shift, upper clamp in the saturating pack
        const int sh = a.shift - 32;
        const long long kadd = (1LL << (a.shift - 1)) - 1;
#pragma unroll
        for (int i = 0; i < G / 16; ++i) {
            uint32_t w[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int b = 16 * i + 4 * j;
                w[j] = pack4_sat(requant8_lo(t[b], kadd, sh), requant8_lo(t[b + 1], kadd, sh),
                                 requant8_lo(t[b + 2], kadd, sh), requant8_lo(t[b + 3], kadd, sh));
            }
            reinterpret_cast<int4 *>(row + col)[i] = make_int4((int)w[0], (int)w[1], (int)w[2], (int)w[3]);
        }
        return;
    }
#pragma unroll
    for (int i = 0; i < G / 16; ++i) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int b = 16 * i + 4 * j;
            w[j] = pack4(requant8(t[b], a.shift), requant8(t[b + 1], a.shift), requant8(t[b + 2], a.shift),
                         requant8(t[b + 3], a.shift));
        }
        reinterpret_cast<int4 *>(row + col)[i] = make_int4((int)w[0], (int)w[1], (int)w[2], (int)w[3]);
    }
}
// Codes already in [-127, 127], written to this thread's row of the output tile.
template <int G>
__device__ __forceinline__ void store_codes_i32(uint8_t *row, int col, const int (&x)[G]) {
#pragma unroll
    for (int i = 0; i < G / 16; ++i) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int b = 16 * i + 4 * j;
            w[j] = pack4(x[b], x[b + 1], x[b + 2], x[b + 3]);
        }
        reinterpret_cast<int4 *>(row + col)[i] = make_int4((int)w[0], (int)w[1], (int)w[2], (int)w[3]);
    }
}

// Float32 output goes straight to global memory (no shared-memory staging).
template <int G>
__device__ __forceinline__ void store_f32(float *gout, int col, const float (&t)[G]) {
    if (!gout) return;
#pragma unroll
    for (int i = 0; i < G / 4; ++i)
        reinterpret_cast<float4 *>(gout + col)[i] = make_float4(t[4 * i], t[4 * i + 1], t[4 * i + 2], t[4 * i + 3]);
}

__device__ __forceinline__ long long relu(long long v) { return ((int)(v >> 32)) < 0 ? 0LL : v; }
__device__ __forceinline__ float relu(float v) { return fmaxf(v, 0.f); }

// One group of G <= 64 columns held entirely in registers.
template <int G>
__device__ __forceinline__ void epi_group(const EpiCtx &e, const ConvArgs &a, int col) {
    if (a.general) {
        // Sec. general nonlinearities: z = clamp(round(H~_out (M_out (.) a) / 2^n_out)),
        // u = phi_int(z), x = clamp(round(H~_next (M_in u) / 2^n_in)); |H~_next u| <= 127 * 64
        // fits int32 and M_in is one scalar, so the next transform runs on u itself
        long long t[G];
#pragma unroll
        for (int q = 0; q < G / 16; ++q) {
            int v[16];
            load_acc16(e, col + 16 * q, v);
            scale_i64(e, col + 16 * q, v, t + 16 * q);
        }
        if (a.hb_out) fwht<G>(t, a.hb_out);
        int u[G];
#pragma unroll
        for (int i = 0; i < G; ++i) u[i] = (int)e.lut[requant8_any(t[i], a.shift) + 127];
        if (a.hb_next) fwht<G>(u, a.hb_next);
        int x[G];
#pragma unroll
        for (int i = 0; i < G; ++i) x[i] = requant8_any(a.mult_in * (long long)u[i], a.shift_in);
        store_codes_i32<G>(e.row, col, x);
        return;
    }
    if (!a.out_f32) {
        long long t[G];
#pragma unroll
        for (int q = 0; q < G / 16; ++q) {
            int v[16];
            load_acc16(e, col + 16 * q, v);
            scale_i64(e, col + 16 * q, v, t + 16 * q);
        }
        if (a.hb_out) fwht<G>(t, a.hb_out);
        if (a.act) {
#pragma unroll
            for (int i = 0; i < G; ++i) t[i] = relu(t[i]);
        }
        if (a.hb_next) fwht<G>(t, a.hb_next);
        store_codes<G>(a, e.row, col, t);
    } else {
        float t[G];
#pragma unroll
        for (int q = 0; q < G / 16; ++q) {
            int v[16];
            load_acc16(e, col + 16 * q, v);
            scale_f32(e, col + 16 * q, v, t + 16 * q);
        }
        if (a.hb_out) fwht<G>(t, a.hb_out);
        if (a.act) {
#pragma unroll
            for (int i = 0; i < G; ++i) t[i] = relu(t[i]);
        }
        store_f32<G>(e.gout, col, t);
    }
}

// A 128-column group (n_t = 128, nbuf = 1) shared by the two epilogue
// warpgroups: warpgroup wg produces outputs 64 wg .. 64 wg + 63 of the
// transition of Eq. integer_hadamard_transition.
//   before phi: p = H~_out (M (.) a) on this half. For hb_out = 128,
//     H~_128 [t_lo; t_hi] = [H~_64 (t_lo + t_hi); H~_64 (t_lo - t_hi)]
//     (both halves of the accumulator are read); smaller blocks lie inside
//     the half.
//   after phi: for hb_next = 128 the two halves u_0, u_1 of phi(p) are
//     exchanged through shared memory (eight int64 per thread and round)
//     and H~_128 [u_0; u_1] = [H~_64 (u_0 + u_1); H~_64 (u_0 - u_1)] gives
//     this half; smaller blocks again lie inside the half.
// One round-shift at the end, as in every other group. Every thread of both
// warpgroups runs the integer path with its exchange barriers, also after an
// abort (ok false: the values are then meaningless but stay in this CTA's
// tensor and shared memory, and the copy-out is skipped), so the named
// barrier always completes.
__device__ __forceinline__ void epi_split128(const EpiCtx &e, const ConvArgs &a, int wg, bool ok, uint8_t *xbuf,
                                             int row) {
    const int half = 64 * wg;
    if (a.out_f32) {
        if (!ok) return;
        float p[64];
        if (a.hb_out == 128) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                int v[16];
                float x[16];
                load_acc16(e, 16 * q, v);
                scale_f32(e, 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) p[16 * q + i] = x[i];
                load_acc16(e, 64 + 16 * q, v);
                scale_f32(e, 64 + 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) p[16 * q + i] = wg ? p[16 * q + i] - x[i] : p[16 * q + i] + x[i];
            }
            fwht_fixed<64, 64>(p);
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                int v[16];
                load_acc16(e, half + 16 * q, v);
                scale_f32(e, half + 16 * q, v, p + 16 * q);
            }
            if (a.hb_out) fwht<64>(p, a.hb_out);
        }
        if (a.act) {
#pragma unroll
            for (int i = 0; i < 64; ++i) p[i] = relu(p[i]);
        }
        store_f32<64>(e.gout, half, p);
        return;
    }
    long long p[64];
    if (a.hb_out == 128) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int v[16];
            long long x[16];
            load_acc16(e, 16 * q, v);
            scale_i64(e, 16 * q, v, x);
#pragma unroll
            for (int i = 0; i < 16; ++i) p[16 * q + i] = x[i];
            load_acc16(e, 64 + 16 * q, v);
            scale_i64(e, 64 + 16 * q, v, x);
#pragma unroll
            for (int i = 0; i < 16; ++i) p[16 * q + i] = wg ? p[16 * q + i] - x[i] : p[16 * q + i] + x[i];
        }
        fwht_fixed<64, 64>(p);
    } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int v[16];
            load_acc16(e, half + 16 * q, v);
            scale_i64(e, half + 16 * q, v, p + 16 * q);
        }
        if (a.hb_out) fwht<64>(p, a.hb_out);
    }
    if (a.act) {
#pragma unroll
        for (int i = 0; i < 64; ++i) p[i] = relu(p[i]);
    }
    if (a.hb_next == 128) {
        // [warpgroup][pair k][row] in 16-byte units: a warp's accesses are 512 contiguous bytes
        int4 *mine = reinterpret_cast<int4 *>(xbuf) + wg * 512 + row;
        const int4 *theirs = reinterpret_cast<const int4 *>(xbuf) + (wg ^ 1) * 512 + row;
#pragma unroll
        for (int r = 0; r < 8; ++r) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const long long u0 = p[8 * r + 2 * k], u1 = p[8 * r + 2 * k + 1];
                mine[k * 128] = make_int4((int)u0, (int)(u0 >> 32), (int)u1, (int)(u1 >> 32));
            }
            asm volatile("bar.sync 4, 256;" ::: "memory");
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int4 v = theirs[k * 128];
                const long long o0 = (long long)(((unsigned long long)(uint32_t)v.y << 32) | (uint32_t)v.x);
                const long long o1 = (long long)(((unsigned long long)(uint32_t)v.w << 32) | (uint32_t)v.z);
                const int i0 = 8 * r + 2 * k;
                p[i0] = wg ? o0 - p[i0] : p[i0] + o0;               // u_0 - u_1 on the upper half, u_0 + u_1 on the lower
                p[i0 + 1] = wg ? o1 - p[i0 + 1] : p[i0 + 1] + o1;
            }
            asm volatile("bar.sync 4, 256;" ::: "memory");
        }
        fwht_fixed<64, 64>(p);
    } else if (a.hb_next) {
        fwht<64>(p, a.hb_next);
    }
    store_codes<64>(a, e.row, half, p);
}

// ------------------------------------------------------------------ kernel

// One CTA per SM, looping over output tiles (tile t -> M tile t / n_tiles_n,
// N tile t % n_tiles_n). The stage ring runs continuously across tiles. TMEM
// holds two fp32 accumulator regions and the reduction runs in exact chunks
// of at most 1024 (sums below 2^24), chunk g accumulating in region g & 1, so
// the MMA issuer fills one region while the epilogue empties the other. With
// one chunk per tile epilogue warpgroup w takes the tiles of region w; with
// several, both warpgroups drain every chunk into int32 register partials
// (half of the 32-column groups each) and finish the tile together.
// SUB: 64-wide reduction blocks per pipeline stage (1, 2 or 4). PIECES: the
// activation blocks arrive as two 32-channel boxes (c % 64 == 32); a separate
// instantiation, so that the other layers' kernels carry none of its code.
template <int SUB, bool PIECES>
__global__ void __launch_bounds__(kThreads, 1)
    conv_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ ConvArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = a.stages;
    uint8_t *staging = smem + (size_t)S * a.stage_bytes;
    uint8_t *bar_area = staging + (size_t)a.staging_bytes;
    const uint32_t bar0 = smem_addr(bar_area);
    // barriers: full[S], conv[S], empty[S], acc_full[2], acc_empty[2], a_free[4], mma_done
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto conv_bar = [&](int s) { return bar0 + 8u * (S + s); };
    auto empty_bar = [&](int s) { return bar0 + 8u * (2 * S + s); };
    auto acc_full = [&](int b) { return bar0 + 8u * (3 * S + b); };
    auto acc_empty = [&](int b) { return bar0 + 8u * (3 * S + 2 + b); };
    auto a_free = [&](int q) { return bar0 + 8u * (3 * S + 4 + q); };
    const uint32_t mma_done = bar0 + 8u * (3 * S + 8);
    // small-channel layers with a TMA-loaded input window: two window buffers
    auto win_full = [&](int b) { return bar0 + 8u * (3 * S + 9 + b); };
    auto win_empty = [&](int b) { return bar0 + 8u * (3 * S + 11 + b); };
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_area + 8 * (3 * S + 13));
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_area + 8 * (3 * S + 13) + 4);

    // A failure already recorded by this launch (or an earlier, unread one)
    // ends every CTA that has not started, so a fault cannot serialize waits.
    // One thread reads the word so the whole CTA takes the same decision.
    __shared__ int s_skip;
    if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int *>(a.err);
    __syncthreads();
    if (s_skip != 0) return;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int tiles_per_img = a.tiles_w * a.tiles_h;
    // nbuf == 2: the epilogue warpgroups alternate tiles, each taking all columns;
    // nbuf == 1 (reduction in several exact chunks): both warpgroups take every
    // chunk, each for half of the 32-column groups, and keep the int32 partial
    // sums of their columns in registers.
    const int nbuf = a.nbuf;
    const int ep_count = nbuf == 2 ? 128 : 256;     // epilogue threads that release a region

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(conv_bar(s), kConvThreads);
            mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(acc_full(b), 1);
            mbar_init(acc_empty(b), ep_count);
        }
        for (int q = 0; q < 4; ++q) mbar_init(a_free(q), 1);
        mbar_init(mma_done, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(win_full(b), 1);
            mbar_init(win_empty(b), kConvThreads);
        }
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_holder)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // bias codes, multipliers and dequant factors of all output channels,
    // staged once per CTA (128-byte aligned, read with 16-byte vector loads)
    int *cb = reinterpret_cast<int *>(bar_area + a.const_off);
    const float s_aff = a.affine ? *a.affine_s : 0.f;
    for (int c = threadIdx.x; c < a.co; c += kThreads) {
        cb[c] = a.b_int[c];
        cb[a.co + c] = a.mult[c];
        reinterpret_cast<float *>(cb)[2 * a.co + c] = a.affine ? s_aff * a.s_w[c] * a.inv_gamma : a.deq[c];
        reinterpret_cast<float *>(cb)[3 * a.co + c] = a.affine ? a.deq[c] : 0.f;
    }
    int8_t *lut_s = reinterpret_cast<int8_t *>(bar_area + a.lut_off);
    if (a.general)
        for (int i = threadIdx.x; i < 256; i += kThreads) lut_s[i] = a.lut[i];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;

    const int nchunks = (a.num_kb + a.chunk_kb - 1) / a.chunk_kb;
    const int my_tiles = a.num_tiles > (int)blockIdx.x ? (a.num_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
    auto tile_coords = [&](int j, int &img, int &ho0, int &wo0, int &n0) {
        const int t = (int)blockIdx.x + j * (int)gridDim.x;
        const int mt = t / a.n_tiles_n;
        n0 = (t - mt * a.n_tiles_n) * a.n_t;
        img = mt / tiles_per_img;
        const int rem = mt - img * tiles_per_img;
        const int ty = rem / a.tiles_w;
        ho0 = ty * a.th;
        wo0 = (rem - ty * a.tiles_w) * a.tw;
    };

    // Register split by warpgroup (launch: 512 x 128 = 65536): warpgroup 0
    // (producer, MMA issuer, two idle warps) 40, warpgroup 3 (converters) 72,
    // warpgroups 1-2 (epilogue) 200: 128 x (40 + 72) + 256 x 200 = 65536, and
    // per scheduler (one warp of each warpgroup) 32 x (40 + 72 + 2 x 200) = 16384.
    const int SA = a.a_slots;
    if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 40;" ::: "memory");
    if (warp == 0) {
        // ---------------------------------------------------------- TMA producer
        if (lane == 0) {
            // stage s with phase parity ph, advanced incrementally (the issuing
            // threads of the pipeline avoid integer division)
            const uint32_t tx_bytes = (uint32_t)(a.b_bytes + (a.gather ? 0 : a.raw_bytes));
            int issued_ph[8];
            for (int q = 0; q < 8; ++q) issued_ph[q] = -1;
            int win_ph[2] = {-1, -1};
            bool ok = true;
            int s = 0;
            uint32_t ph = 0;
            for (int j = 0; j < my_tiles && ok; ++j) {
                int img, ho0, wo0, n0;
                tile_coords(j, img, ho0, wo0, n0);
                if (a.win_tma) {
                    // the tile's input window: one 3-D box of the [n][h][w c] byte tensor, its first byte
                    // column rounded down to 16 (out-of-image parts, also negative ones, are zero-filled)
                    const int b = j & 1;
                    if (j >= 2 && !mbar_wait(win_empty(b), ((j >> 1) - 1) & 1, abort_flag, a.err)) { ok = false; break; }
                    mbar_expect_tx(win_full(b), (uint32_t)a.win_tma_bytes);
                    const int xb = (wo0 * a.stride - a.pad_x) * a.c;
                    tma_load_3d(smem_addr(bar_area + a.win_off + b * a.win_buf), &tmA, win_full(b), xb & ~15,
                                ho0 * a.stride - a.pad_y, img);
                    win_ph[b] = (j >> 1) & 1;
                }
                int cb = 0, kx = 0, ky = 0;          // 64-channel block, kernel column and row of block kb
                for (int kb0 = 0; kb0 < a.num_kb; kb0 += SUB) {
                    const int nsub = min(SUB, a.num_kb - kb0);
                    if (!mbar_wait(empty_bar(s), ph ^ 1, abort_flag, a.err)) { ok = false; break; }
                    const uint32_t st = smem_addr(smem + (size_t)s * a.stage_bytes);
                    mbar_expect_tx(full_bar(s), tx_bytes * (uint32_t)nsub);
#pragma unroll
                    for (int u = 0; u < SUB; ++u) {
                        if (u >= nsub) break;
                        tma_load_2d(st + a.b_off + u * a.b_bytes, &tmB, full_bar(s), (kb0 + u) * kBlockK, n0);
                        if constexpr (!PIECES) {
                            if (!a.gather) {
                                tma_load_4d(st + a.raw_off + u * a.raw_bytes, &tmA, full_bar(s), cb * kBlockK,
                                            wo0 * a.stride + kx - a.pad_x, ho0 * a.stride + ky - a.pad_y, img);
                                if (++cb == a.cin_kb) {
                                    cb = 0;
                                    if (++kx == a.kw) { kx = 0; ++ky; }
                                }
                            }
                        } else {
                            // two 32-channel pieces (cb counts pieces); past the last tap the
                            // weights are zero and the box, in or out of the image, is read as is
#pragma unroll
                            for (int hp = 0; hp < 2; ++hp) {
                                tma_load_4d(st + a.raw_off + u * a.raw_bytes + hp * (a.raw_bytes >> 1), &tmA,
                                            full_bar(s), cb * 32, wo0 * a.stride + kx - a.pad_x,
                                            ho0 * a.stride + ky - a.pad_y, img);
                                if (++cb == a.cin_h) {
                                    cb = 0;
                                    if (++kx == a.kw) { kx = 0; ++ky; }
                                }
                            }
                        }
                    }
                    issued_ph[s] = (int)ph;
                    if (++s == S) { s = 0; ph ^= 1u; }
                }
            }
            if (!ok) {
                // let our own copies land before the CTA unwinds
                for (int b = 0; b < 2; ++b)
                    if (win_ph[b] >= 0) {
                        const long long t0 = clock64();
                        while (!mbar_try_wait(win_full(b), (uint32_t)win_ph[b]) && clock64() - t0 < kWaitLimitCycles) {
                        }
                    }
                for (int q = 0; q < S && q < 8; ++q)
                    if (issued_ph[q] >= 0) {
                        const long long t0 = clock64();
                        while (!mbar_try_wait(full_bar(q), (uint32_t)issued_ph[q]) && clock64() - t0 < kWaitLimitCycles) {
                        }
                    }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16(a.n_t);
            // weight descriptor of stage 0, block 0; a stage / block moves its start address field
            const uint64_t desc0 = sdesc_sw128(smem_addr(smem) + (uint32_t)a.b_off);
            // fp16 operand codes: the A tile of the stage (128 rows of 128 bytes per block, 128-byte swizzle)
            const uint64_t adesc0 = sdesc_sw128(smem_addr(smem) + (uint32_t)a.raw_off);
            const uint32_t stage_step = (uint32_t)a.stage_bytes >> 4, blk_step = (uint32_t)a.b_bytes >> 4;
            const uint32_t raw_step = (uint32_t)a.raw_bytes >> 4;
            const bool a_f16 = a.a_f16 != 0;
            bool ok = true;
            int s = 0, slot = 0;
            uint32_t ph = 0;
            int g = 0;                       // exact chunks issued so far; chunk g accumulates in region g & 1
            uint32_t d_tmem = tmem;
            for (int j = 0; j < my_tiles && ok; ++j) {
                // a stage holds SUB 64-wide reduction blocks; chunk boundaries
                // (multiples of chunk_kb, itself a multiple of SUB) fall between stages
                int ck = 0;                  // blocks of the current exact chunk already issued
                for (int kb0 = 0; kb0 < a.num_kb; kb0 += SUB) {
                    const int nsub = min(SUB, a.num_kb - kb0);
                    if (ck == 0) {
                        d_tmem = tmem + (uint32_t)((g & 1) * a.n_t);
                        if (g >= 2) {        // wait until the epilogue released the region
                            if (!mbar_wait(acc_empty(g & 1), ((g >> 1) - 1) & 1, abort_flag, a.err)) { ok = false; break; }
                            tc_fence_after();
                        }
                    }
                    // conv[s] completes only after every converter observed full[s] (the TMA
                    // bytes of this stage), so waiting for it orders the weight reads as well
                    if (!mbar_wait(conv_bar(s), ph, abort_flag, a.err)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t db0 = desc0 + (uint64_t)((uint32_t)s * stage_step);
                    if (!a_f16) {
                        const uint32_t a_t = tmem + (uint32_t)(a.a_col + slot * SUB * 32);
#pragma unroll
                        for (int u = 0; u < SUB; ++u) {
                            if (u >= nsub) break;
                            const uint64_t db = db0 + (uint64_t)((uint32_t)u * blk_step);
#pragma unroll
                            for (int kk = 0; kk < kBlockK / 16; ++kk)   // K = 16 per instruction: 8 TMEM columns, 32 bytes of B
                                umma_f16_ts(d_tmem, a_t + (uint32_t)(u * 32 + kk * 8), db + (uint64_t)(2 * kk), idesc,
                                            (ck + u > 0 || kk > 0) ? 1u : 0u);
                        }
                    } else {
                        const uint64_t da0 = adesc0 + (uint64_t)((uint32_t)s * stage_step);
#pragma unroll
                        for (int u = 0; u < SUB; ++u) {
                            if (u >= nsub) break;
                            const uint64_t db = db0 + (uint64_t)((uint32_t)u * blk_step);
                            const uint64_t da = da0 + (uint64_t)((uint32_t)u * raw_step);
#pragma unroll
                            for (int kk = 0; kk < kBlockK / 16; ++kk)   // both operands in shared memory, 32 bytes each
                                umma_f16_ss(d_tmem, da + (uint64_t)(2 * kk), db + (uint64_t)(2 * kk), idesc,
                                            (ck + u > 0 || kk > 0) ? 1u : 0u);
                        }
                    }
                    umma_commit(empty_bar(s));
                    umma_commit(a_free(slot));
                    ck += nsub;
                    if (ck == a.chunk_kb || kb0 + nsub == a.num_kb) {
                        umma_commit(acc_full(g & 1));
                        ++g;
                        ck = 0;
                    }
                    if (++s == S) { s = 0; ph ^= 1u; }
                    if (++slot == SA) slot = 0;
                }
            }
            umma_commit(mma_done);
            const long long t0 = clock64();
            while (!mbar_try_wait(mma_done, 0) && clock64() - t0 < kWaitLimitCycles) {
            }
        }
    }
    } else if (warp >= 12) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 72;" ::: "memory");
        // ---------------------------------------------------------- converters (warps 12-15)
        // Thread m converts row m of the A operand (output pixel m of the tile)
        // into TMEM lane m: 64 INT8 codes -> 32 columns of fp16 pairs.
        const int quad = warp & 3;
        const int m = quad * 32 + lane;               // 0..127
        const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)a.a_col;
        bool ok = true;
        // stage s (phase parity ph) and A slot (use parity sph), advanced incrementally
        int s = 0, slot = 0;
        uint32_t ph = 0, sph = 0;
        bool reuse = false;                           // the slot was used before (some slot wrapped)
        auto advance = [&]() {
            if (++s == S) { s = 0; ph ^= 1u; }
            if (++slot == SA) { slot = 0; sph ^= 1u; reuse = true; }
        };
        // wait until the A slot was released by the MMAs that last read it
        auto slot_free = [&]() {
            bool w = !reuse || mbar_wait(a_free(slot), sph ^ 1u, abort_flag, a.err);
            w = __all_sync(0xffffffffu, w);
            tc_fence_after();
            return w;
        };
        if (!a.gather) {
            // row m of a 64-wide INT8 box (64 bytes, 16-byte chunks permuted by the
            // 64-byte swizzle) -> 32 columns of fp16 pairs
            auto convert_row = [&](const uint8_t *raw, uint32_t (&h)[32]) {
                if (a.affine) {
                    // row m of a 64-wide int16 box (128 bytes, 16-byte chunks permuted by the 128-byte
                    // swizzle), or of two 32-wide boxes (64-byte rows, 64-byte swizzle)
                    const int sw = PIECES ? (m >> 1) & 3 : m & 7;
                    const int hb = a.raw_bytes >> 1;
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int off = PIECES ? (q >> 2) * hb + (((q & 3) ^ sw) << 4) : (q ^ sw) << 4;
                        const uint4 v = *reinterpret_cast<const uint4 *>(raw + off);
                        h[4 * q + 0] = i16x2_to_f16x2(v.x);
                        h[4 * q + 1] = i16x2_to_f16x2(v.y);
                        h[4 * q + 2] = i16x2_to_f16x2(v.z);
                        h[4 * q + 3] = i16x2_to_f16x2(v.w);
                    }
                    return;
                }
                uint4 v[4];
                if constexpr (PIECES) {
                    // two 32-wide boxes: 32-byte rows, chunk pairs swapped by the 32-byte swizzle
                    const int sw = (m >> 2) & 1;
                    const int hb = a.raw_bytes >> 1;
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        v[q] = *reinterpret_cast<const uint4 *>(raw + (q >> 1) * hb + (((q & 1) ^ sw) << 4));
                } else {
                    const int sw = (m >> 1) & 3;
#pragma unroll
                    for (int q = 0; q < 4; ++q) v[q] = *reinterpret_cast<const uint4 *>(raw + ((q ^ sw) << 4));
                }
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    i8x4_to_f16x4(v[q].x, h[8 * q + 0], h[8 * q + 1]);
                    i8x4_to_f16x4(v[q].y, h[8 * q + 2], h[8 * q + 3]);
                    i8x4_to_f16x4(v[q].z, h[8 * q + 4], h[8 * q + 5]);
                    i8x4_to_f16x4(v[q].w, h[8 * q + 6], h[8 * q + 7]);
                }
            };
            // bytes of one operand row of a 64-wide block (of one of its 32-wide boxes with a.half)
            const int row_in = ((a.affine || a.a_f16) ? 128 : 64) >> (PIECES ? 1 : 0);
            for (int j = 0; j < my_tiles && ok; ++j) {
                for (int kb0 = 0; kb0 < a.num_kb; kb0 += SUB) {
                    const int nsub = min(SUB, a.num_kb - kb0);
                    ok = __all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, abort_flag, a.err));
                    if (!ok) break;
                    const uint8_t *raw = smem + (size_t)s * a.stage_bytes + a.raw_off + m * row_in;
                    const uint32_t t_slot = t_lane + (uint32_t)(slot * SUB * 32);
                    if (a.a_f16) {
                        // the MMAs read the fp16 tile itself; only the hand-off remains
                        ok = slot_free();
                        if (!ok) break;
                        tc_fence_before();
                        mbar_arrive(conv_bar(s));
                        advance();
                        continue;
                    }
                    uint32_t h[32];
                    convert_row(raw, h);              // the first block is converted before the slot frees up
                    ok = slot_free();
                    if (!ok) break;
                    tmem_st32(t_slot, h);
#pragma unroll 1
                    for (int u = 1; u < SUB; ++u) {
                        if (u >= nsub) break;
                        convert_row(raw + u * a.raw_bytes, h);
                        tmem_st32(t_slot + (uint32_t)(u * 32), h);
                    }
                    tmem_wait_st();
                    tc_fence_before();
                    mbar_arrive(conv_bar(s));
                    advance();
                }
            }
        } else {
            // Small-channel layer. Each tile's input window ((th-1)s+kh rows of
            // (tw-1)s+kw pixels, zero outside the image) is copied to shared
            // memory; kernel row ky of output pixel m is then one contiguous
            // kw*c-byte segment of window row py*s+ky, read as 8-entry pieces
            // through a per-CTA table (window offset of each piece, -1 = zero).
            int *tab = reinterpret_cast<int *>(bar_area + 8 * (3 * S + 13) + 16);
            uint8_t *win = bar_area + a.win_off;
            for (int q = m; q < a.num_kb * 8; q += kConvThreads) {
                const int k0 = q * 8, ky = k0 / a.seg;
                tab[q] = ky < a.kh ? ky * a.win_pitch + (k0 - ky * a.seg) : -1;
            }
            const int rbase = (m / a.tw) * a.stride * a.win_pitch + (m % a.tw) * a.stride * a.c;
            // Without a TMA window, every converter thread runs the same tile loop
            // (also after an abort, doing no work) so all four warps reach each named
            // barrier. With one (win_tma) the producer loads the window one tile
            // ahead into one of two buffers and no named barrier is used.
            for (int j = 0; j < my_tiles; ++j) {
                int img, ho0, wo0, n0;
                tile_coords(j, img, ho0, wo0, n0);
                const uint8_t *wv = win;                  // this tile's window
                int woff = 0;                             // its first byte inside the buffer
                if (a.win_tma) {
                    if (!ok) break;
                    const int b = j & 1;
                    ok = __all_sync(0xffffffffu, mbar_wait(win_full(b), (j >> 1) & 1, abort_flag, a.err));
                    if (!ok) break;
                    wv = win + b * a.win_buf;
                    const int xb = (wo0 * a.stride - a.pad_x) * a.c;
                    woff = xb - (xb & ~15);
                }
                if (!a.win_tma) asm volatile("bar.sync 1, %0;" ::"r"(kConvThreads) : "memory");   // previous window consumed
                if (ok && !a.win_tma) {
                    const int ix_lo = wo0 * a.stride - a.pad_x;
                    const int row_b = a.win_w * a.c;
                    const int b_lo = max(0, -ix_lo) * a.c, b_hi = min(a.win_w, a.w - ix_lo) * a.c;
                    // per row, all of a thread's loads are issued before its stores
                    for (int r = 0; r < a.win_h; ++r) {
                        const int iy = ho0 * a.stride - a.pad_y + r;
                        const bool row_in = iy >= 0 && iy < a.h;
                        const int8_t *src = a.x + (((long long)img * a.h + (row_in ? iy : 0)) * a.w + ix_lo) * a.c;
                        for (int b0 = m; b0 < row_b; b0 += 8 * kConvThreads) {
                            uint8_t v[8];
#pragma unroll
                            for (int u = 0; u < 8; ++u) {
                                const int b = b0 + u * kConvThreads;
                                v[u] = (row_in && b >= b_lo && b < b_hi) ? (uint8_t)__ldg(src + b) : (uint8_t)0;
                            }
#pragma unroll
                            for (int u = 0; u < 8; ++u) {
                                const int b = b0 + u * kConvThreads;
                                if (b < row_b) win[r * a.win_pitch + b] = v[u];
                            }
                        }
                    }
                }
                if (!a.win_tma) asm volatile("bar.sync 1, %0;" ::"r"(kConvThreads) : "memory");   // window complete
                for (int kb = 0; kb < a.num_kb && ok; ++kb) {
                    // the operand comes from the window: it is built first, then the
                    // stage (which keeps conv[s] in step with the MMA issuer) and the
                    // A slot are waited for
                    uint32_t h[32];
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int off = tab[kb * 8 + q];
                        uint32_t w0 = 0u, w1 = 0u;
                        if (off >= 0) {
                            const int o = rbase + woff + off;
                            const uint32_t *p = reinterpret_cast<const uint32_t *>(wv + (o & ~3));
                            const uint32_t x0 = p[0], x1 = p[1], x2 = p[2];
                            w0 = __funnelshift_r(x0, x1, (uint32_t)(o & 3) * 8u);
                            w1 = __funnelshift_r(x1, x2, (uint32_t)(o & 3) * 8u);
                        }
                        i8x4_to_f16x4(w0, h[4 * q + 0], h[4 * q + 1]);
                        i8x4_to_f16x4(w1, h[4 * q + 2], h[4 * q + 3]);
                    }
                    ok = __all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, abort_flag, a.err));
                    if (!ok) break;
                    ok = slot_free();
                    if (!ok) break;
                    tmem_st32(t_lane + (uint32_t)(slot * 32), h);
                    tmem_wait_st();
                    tc_fence_before();
                    mbar_arrive(conv_bar(s));
                    advance();
                }
                if (a.win_tma && ok) mbar_arrive(win_empty(j & 1));   // this thread's reads of the window are done
            }
        }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 200;" ::: "memory");
        // ---------------------------------------------------------- epilogue warpgroups (warps 4-7, 8-11)
        const int wg = (warp - 4) >> 2;            // 0 or 1
        const int quad = warp & 3;                 // TMEM lane quadrant this warp may access
        const int row = quad * 32 + lane;
        const int et = threadIdx.x - 128 - 128 * wg;   // 0..127 within the warpgroup
        const int esz = a.out_f32 ? 4 : 1;
        const int row_bytes = a.n_t * esz;
        uint8_t *stage_tile = staging + (size_t)(nbuf == 2 ? wg : 0) * kTileM * a.row_stride;
        const int G = max(32, max(a.hb_out, a.hb_next));
        uint32_t part[4][32];                      // nbuf == 1: int32 partial sums of column groups 2k + wg
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int i = 0; i < 32; ++i) part[k][i] = 0u;
        bool ok = true;
        // Every epilogue thread runs the same loops (also after an abort, doing
        // no work) so the warpgroups reach each named barrier together.
        for (int j = 0; j < my_tiles; ++j) {
            if (nbuf == 2 && (j & 1) != wg) continue;
            int img, ho0, wo0, n0;
            tile_coords(j, img, ho0, wo0, n0);
            for (int ch = 0; ch < nchunks; ++ch) {
                const int g = j * nchunks + ch;    // chunk index, as counted by the MMA issuer
                const int reg = g & 1;
                const uint32_t t_acc = tmem + (uint32_t)(reg * a.n_t) + ((uint32_t)(quad * 32) << 16);
                if (ok) {
                    ok = __all_sync(0xffffffffu, mbar_wait(acc_full(reg), (g >> 1) & 1, abort_flag, a.err));
                    tc_fence_after();
                }
                if (ch + 1 < nchunks) {
                    // drain: chunk sum -> register partials; the region goes straight back to the MMA issuer
                    if (ok) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int col = (2 * k + wg) * 32;
                            if (col >= a.n_t) break;
                            uint32_t r[32];
                            tmem_ld32(t_acc + col, r);
                            tmem_wait_ld();
#pragma unroll
                            for (int i = 0; i < 32; ++i) part[k][i] += (uint32_t)__float2int_rn(__uint_as_float(r[i]));
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(acc_empty(reg));
                    continue;
                }
                if (nbuf == 1) {
                    // last chunk: chunk sum + partial -> exact int32 totals, written back in place so
                    // that each 64/128-wide transform group can read all of its columns
                    if (ok) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int col = (2 * k + wg) * 32;
                            if (col >= a.n_t) break;
                            uint32_t r[32];
                            tmem_ld32(t_acc + col, r);
                            tmem_wait_ld();
#pragma unroll
                            for (int i = 0; i < 32; ++i) r[i] = part[k][i] + (uint32_t)__float2int_rn(__uint_as_float(r[i]));
                            tmem_st32(t_acc + col, r);
                        }
                        tmem_wait_st();
                    }
                    tc_fence_before();
                    asm volatile("bar.sync 4, 256;" ::: "memory");
                    tc_fence_after();
                }
                // the partials restart at zero for the next tile (and are dead during the groups)
#pragma unroll
                for (int k = 0; k < 4; ++k)
#pragma unroll
                    for (int i = 0; i < 32; ++i) part[k][i] = 0u;
                EpiCtx e;
                e.b_int = cb + n0;
                e.mult = cb + a.co + n0;
                e.deq = reinterpret_cast<const float *>(cb + 2 * a.co) + n0;
                e.biasf = reinterpret_cast<const float *>(cb + 3 * a.co) + n0;
                e.t_acc = t_acc;
                e.int_acc = nbuf == 1;
                e.lut = lut_s;
                e.row = stage_tile + (size_t)row * a.row_stride;
                e.gout = nullptr;
                if (a.out_f32) {
                    const int oy = ho0 + row / a.tw, ox = wo0 + row % a.tw;
                    if (oy < a.ho && ox < a.wo)
                        e.gout = static_cast<float *>(a.y) + (((long long)img * a.y_h + oy * a.ostride + a.ooy) * a.y_w +
                                                              ox * a.ostride + a.oox) * a.co + n0;
                }
                if (G == 128) {
                    // n_t == 128, nbuf == 1: the warpgroups share the group; the shared-memory
                    // output tile is free until the codes are stored and serves as the exchange buffer
                    epi_split128(e, a, wg, ok, stage_tile, row);
                } else if (ok) {
                    int gi = 0;
                    for (int col = 0; col < a.n_t; col += G, ++gi) {
                        if (nbuf == 1 && (gi & 1) != wg) continue;
                        if (G == 32) epi_group<32>(e, a, col);
                        else epi_group<64>(e, a, col);
                    }
                }
                tc_fence_before();
                mbar_arrive(acc_empty(reg));           // TMEM reads of this region are complete
                // coalesced copy-out: consecutive threads write consecutive 16-byte chunks
                const int nthr = nbuf == 2 ? 128 : 256;
                const int tid = nbuf == 2 ? et : et + 128 * wg;
                if (nbuf == 2) asm volatile("bar.sync %0, 128;" ::"r"(2 + wg) : "memory");
                else asm volatile("bar.sync 4, 256;" ::: "memory");
                // a half-warp per tile row (at most 14 chunks of 16 bytes), so no division per chunk
                const int cpr = row_bytes >> 4;
                const int c = lane & 15;
                for (int r = (tid >> 5) * 2 + (lane >> 4); ok && !a.out_f32 && r < kTileM; r += nthr >> 4) {
                    const int oy = ho0 + (r >> a.tw_log2), ox = wo0 + (r & (a.tw - 1));
                    if (c < cpr && oy < a.ho && ox < a.wo) {
                        const int gy = oy * a.ostride + a.ooy, gx = ox * a.ostride + a.oox;
                        const uint8_t *src = stage_tile + (size_t)r * a.row_stride;
                        if (!a.d2s) {
                            const long long pix = ((long long)img * a.y_h + gy) * a.y_w + gx;
                            const int4 v = *reinterpret_cast<const int4 *>(src + c * 16);
                            if (a.out_f16) {
                                // the same codes as fp16 (exact): 16 codes -> 32 bytes
                                uint32_t hh[8];
                                i8x4_to_f16x4((uint32_t)v.x, hh[0], hh[1]);
                                i8x4_to_f16x4((uint32_t)v.y, hh[2], hh[3]);
                                i8x4_to_f16x4((uint32_t)v.z, hh[4], hh[5]);
                                i8x4_to_f16x4((uint32_t)v.w, hh[6], hh[7]);
                                int4 *dst = reinterpret_cast<int4 *>(static_cast<uint16_t *>(a.y) + pix * a.co + n0 + c * 16);
                                dst[0] = make_int4((int)hh[0], (int)hh[1], (int)hh[2], (int)hh[3]);
                                dst[1] = make_int4((int)hh[4], (int)hh[5], (int)hh[6], (int)hh[7]);
                            } else {
                                *reinterpret_cast<int4 *>(static_cast<uint8_t *>(a.y) + pix * a.co + n0 + c * 16) = v;
                            }
                        } else {
                            // sub-pixel rearrangement: channel cd r^2 + i r + j of pixel (gy, gx) goes to
                            // channel cd of pixel (gy r + i, gx r + j); chunk c holds 16 destination channels
                            // of one (i, j), gathered from the tile row with stride r^2
                            const int rr = a.d2s, r2 = rr * rr, per = cpr / r2;
                            const int g = c / per, q = c - g * per, i = g / rr, j = g - i * rr;
                            const uint8_t *s0 = src + (16 * q) * r2 + i * rr + j;
                            uint32_t wd[4];
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                wd[k] = (uint32_t)s0[(4 * k) * r2] | ((uint32_t)s0[(4 * k + 1) * r2] << 8) |
                                        ((uint32_t)s0[(4 * k + 2) * r2] << 16) | ((uint32_t)s0[(4 * k + 3) * r2] << 24);
                            const int cd = a.co / r2;
                            const long long pix =
                                ((long long)img * a.y_h * rr + gy * rr + i) * ((long long)a.y_w * rr) + gx * rr + j;
                            *reinterpret_cast<int4 *>(static_cast<uint8_t *>(a.y) + pix * cd + n0 / r2 + 16 * q) =
                                make_int4((int)wd[0], (int)wd[1], (int)wd[2], (int)wd[3]);
                        }
                    }
                }
                if (nbuf == 2) asm volatile("bar.sync %0, 128;" ::"r"(2 + wg) : "memory");
                else asm volatile("bar.sync 4, 256;" ::: "memory");
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(a.tmem_cols) : "memory");
    }
}

#if !HATQ_CONV_PIECES
// Failure-detection self test: one thread waits, through the pipeline's
// bounded wait, on an mbarrier nothing arrives at; the wait expires after
// `limit` cycles and records kErrWaitTimeout in the error word.
__global__ void wait_selftest_kernel(int *err, long long limit) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x != 0) return;
    abort_flag = 0;
    mbar_init(smem_addr(&bar), 1);
    fence_barrier_init();
    (void)mbar_wait(smem_addr(&bar), 0, &abort_flag, err, limit);
}

#endif

}  // namespace

#if HATQ_CONV_PIECES
ConvKernelFn conv_pieces_kernel(int sub) {
    return sub == 4 ? conv_kernel<4, true> : (sub == 2 ? conv_kernel<2, true> : conv_kernel<1, true>);
}
#else
cudaError_t launch_wait_selftest(int *err, long long limit_cycles, cudaStream_t s) {
    wait_selftest_kernel<<<1, 32, 0, s>>>(err, limit_cycles);
    return cudaGetLastError();
}

cudaError_t launch_conv(const CUtensorMap &tmA, const CUtensorMap &tmB, const ConvArgs &a, int smem_bytes, cudaStream_t s) {
    // the shared-memory opt-in and the SM count are per device
    constexpr int kMaxDev = 64;
    static int configured_smem[kMaxDev][6] = {};
    static int sms_of[kMaxDev] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
    if ((a.sub != 1 && a.sub != 2 && a.sub != 4) || (a.gather && a.sub != 1) || a.chunk_kb % a.sub ||
        (a.half && (a.gather || a.a_f16 || a.cin_h < 1)))
        return cudaErrorInvalidValue;   // gathered tiles: one block per stage
    const int v = (a.sub == 4 ? 2 : (a.sub == 2 ? 1 : 0)) + (a.half ? 3 : 0);
    const ConvKernelFn kern = a.half ? conv_pieces_kernel(a.sub)
                                     : (v == 2 ? conv_kernel<4, false> : (v == 1 ? conv_kernel<2, false> : conv_kernel<1, false>));
    if (smem_bytes > configured_smem[dev][v]) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return e;
        configured_smem[dev][v] = smem_bytes;
    }
    if (!sms_of[dev]) {
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        sms_of[dev] = sms > 0 ? sms : 1;
    }
    const int grid = a.num_tiles < sms_of[dev] ? a.num_tiles : sms_of[dev];
    kern<<<grid, kThreads, smem_bytes, s>>>(tmA, tmB, a);
    return cudaGetLastError();
}

#endif  // HATQ_CONV_PIECES

}  // namespace hatq
