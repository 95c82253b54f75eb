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
// are exactly representable integers and the chunk sum is exact. After each
// chunk the epilogue warps convert the chunk sum to int32 and add it to an
// int32 partial held in a second TMEM region, so the full accumulator is the
// exact int32 sum.
//
// Warp roles (one 128 x N_t output tile per CTA, 256 threads; two warps per
// SM sub-partition, so each thread may hold up to 255 registers):
//   warp 0     TMA producer: weight tile (fp16, 128B-swizzled) and, for
//              c_in % 16 == 0, the INT8 activation box of one kernel tap and
//              64 input channels (zero fill outside the image = zero padding).
//   warp 1     TMEM allocation; lane 0 issues the MMAs and commits.
//   warps 2-3  converters: INT8 box -> fp16 operand tile in the 128B-swizzled
//              K-major layout the MMA descriptor expects (or, for small c_in,
//              a gather from the tile's input window staged in shared memory).
//   warps 4-7  drain fp32 chunk sums into the int32 partial.
//   all warps  final epilogue once the last MMA completed: warps w and w+4
//              share TMEM lane quadrant w%4 and split the column groups; the
//              output tile is staged in shared memory and copied out coalesced.
// Every mbarrier wait is bounded: on expiry the kernel records an error word,
// raises a CTA-wide abort flag and unwinds (waiting, again bounded, for its own
// MMAs and copies) before freeing TMEM.
#include <cuda_fp16.h>

#include "hatq_internal.h"

namespace hatq {
namespace {

constexpr int kThreads = 256;
constexpr int kConvThreads = 64;       // converter warps 2-3
constexpr int kBlockK = 64;            // fp16 elements per 128-byte swizzle row
constexpr int kTileM = 128;
constexpr long long kWaitLimitCycles = 4000000000LL;   // about 2 s at 2 GHz

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait. Returns false when the CTA aborts (this wait expired, or
// another role raised the abort flag).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag, int *err) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t spin = 1;; ++spin) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((spin & 63) == 0) {
            if (*abort_flag) return false;
            if (*reinterpret_cast<volatile int *>(err) != 0) { *abort_flag = 1; return false; }
            if (clock64() - t0 > kWaitLimitCycles) {
                *abort_flag = 1;
                atomicExch(err, kErrWaitTimeout);
                return false;
            }
        }
    }
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *tm, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"(tm), "r"(bar), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *tm, uint32_t bar, int c0, int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(tm), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

// tcgen05 shared-memory matrix descriptor: K-major operand, 128-byte swizzle,
// 8-row groups 1024 bytes apart (stride byte offset), version field = 1.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;                 // leading byte offset (unused for this layout)
    d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset
    d |= (uint64_t)1 << 46;                 // descriptor version
    d |= (uint64_t)2 << 61;                 // 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::f16: D = f32, A = B = f16, both K-major, M = 128.
__device__ __forceinline__ uint32_t idesc_f16(int n) {
    return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kTileM >> 4) << 24);
}

__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// 32 consecutive TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
        "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

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

// Byte offset of 16-byte chunk `chunk` of row `row` in a 128B-swizzled
// K-major tile (8-row groups of 1024 bytes).
__device__ __forceinline__ uint32_t sw128_offset(int row, int chunk) {
    return (uint32_t)((row >> 3) * 1024 + (row & 7) * 128 + ((chunk ^ (row & 7)) << 4));
}

// ------------------------------------------------------------------ epilogue math

__device__ __forceinline__ int requant8(long long v, int n) {
    // round(v / 2^n) half to even, clamped to [-127, 127]: v + 2^(n-1) - 1 + bit_n(v), then >> n.
    int q;
    if (n >= 32) {
        // |v| < 2^62, so the shifted value fits in 32 bits.
        const long long u = v + ((1LL << (n - 1)) - 1) + ((int)((unsigned long long)v >> n) & 1);
        q = (int)(u >> n);
    } else if (n > 0) {
        const long long u = v + ((1LL << (n - 1)) - 1) + ((v >> n) & 1);
        const long long w = u >> n;
        q = w < -127 ? -127 : (w > 127 ? 127 : (int)w);
    } else {
        q = v < -127 ? -127 : (v > 127 ? 127 : (int)v);
    }
    return q < -127 ? -127 : (q > 127 ? 127 : q);
}

template <int G, int HB, typename T>
__device__ __forceinline__ void fwht_fixed(T (&t)[G]) {
#pragma unroll
    for (int h = 1; h < HB; h <<= 1) {
#pragma unroll
        for (int i = 0; i < G; ++i) {
            if (i & h) continue;
            const T a = t[i], b = t[i + h];
            t[i] = a + b;
            t[i + h] = a - b;
        }
    }
}

// Unnormalized Sylvester transform of every hb-block inside t[0..G).
template <int G, typename T>
__device__ __forceinline__ void fwht(T (&t)[G], int hb) {
    switch (hb) {
        case 2: fwht_fixed<G, 2>(t); break;
        case 4: fwht_fixed<G, 4>(t); break;
        case 8: fwht_fixed<G, 8>(t); break;
        case 16: fwht_fixed<G, 16>(t); break;
        case 32: if (G >= 32) fwht_fixed<G, (G >= 32 ? 32 : 2)>(t); break;
        case 64: if (G >= 64) fwht_fixed<G, (G >= 64 ? 64 : 2)>(t); break;
        default: break;
    }
}

struct EpiCtx {
    const int *b_int;    // this tile's bias codes, multipliers and dequant factors (shared memory)
    const int *mult;
    const float *deq;
    uint32_t t_acc;      // TMEM address of this warp's lanes, column 0 of the accumulator
    uint32_t t_part;     // ... of the int32 partial region
    bool has_part;
    uint8_t *row;        // this thread's row of the shared-memory output tile
};

// Exact int32 accumulator of 16 columns starting at tile column `col`, bias included.
__device__ __forceinline__ void load_acc16(const EpiCtx &e, int col, int (&v)[16]) {
    uint32_t r[16];
    tmem_ld16(e.t_acc + col, r);
    if (e.has_part) {
        uint32_t p[16];
        tmem_ld16(e.t_part + col, p);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = __float2int_rn(__uint_as_float(r[i])) + (int)p[i];
    } else {
        tmem_wait_ld();
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
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float4 d = dp[i];
        t[4 * i] = d.x * (float)v[4 * i];
        t[4 * i + 1] = d.y * (float)v[4 * i + 1];
        t[4 * i + 2] = d.z * (float)v[4 * i + 2];
        t[4 * i + 3] = d.w * (float)v[4 * i + 3];
    }
}

// Requantized codes of G columns starting at tile column col, written to this
// thread's row of the shared-memory output tile (copied out coalesced later).
template <int G>
__device__ __forceinline__ void store_codes(const ConvArgs &a, uint8_t *row, int col, const long long (&t)[G]) {
#pragma unroll
    for (int i = 0; i < G / 16; ++i) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int b = 16 * i + 4 * j;
            w[j] = (uint32_t)(requant8(t[b], a.shift) & 0xff) | ((uint32_t)(requant8(t[b + 1], a.shift) & 0xff) << 8) |
                   ((uint32_t)(requant8(t[b + 2], a.shift) & 0xff) << 16) |
                   ((uint32_t)(requant8(t[b + 3], a.shift) & 0xff) << 24);
        }
        reinterpret_cast<int4 *>(row + col)[i] = make_int4((int)w[0], (int)w[1], (int)w[2], (int)w[3]);
    }
}
template <int G>
__device__ __forceinline__ void store_f32(uint8_t *row, int col, const float (&t)[G]) {
#pragma unroll
    for (int i = 0; i < G / 4; ++i)
        reinterpret_cast<float4 *>(row + 4 * col)[i] = make_float4(t[4 * i], t[4 * i + 1], t[4 * i + 2], t[4 * i + 3]);
}

__device__ __forceinline__ long long relu(long long v) { return ((int)(v >> 32)) < 0 ? 0LL : v; }
__device__ __forceinline__ float relu(float v) { return fmaxf(v, 0.f); }

// One group of G <= 64 columns held entirely in registers.
template <int G>
__device__ __forceinline__ void epi_group(const EpiCtx &e, const ConvArgs &a, int col) {
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
        store_f32<G>(e.row, col, t);
    }
}

// A 128-column group with exactly one 128-wide transform (H~_out or H~_next):
// H~_128 [x_lo; x_hi] = [H~_64 (x_lo + x_hi); H~_64 (x_lo - x_hi)], evaluated
// as two register-resident passes of 64 outputs each.
__device__ __forceinline__ void epi_group128(const EpiCtx &e, const ConvArgs &a, int col) {
    const bool pre_relu = a.act && a.hb_out == 0;     // phi before H~_next
    const bool post_relu = a.act && a.hb_out != 0;    // phi after H~_out
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
        if (!a.out_f32) {
            long long s[64];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                int v[16];
                long long x[16];
                load_acc16(e, col + 16 * q, v);
                scale_i64(e, col + 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) s[16 * q + i] = pre_relu ? relu(x[i]) : x[i];
                load_acc16(e, col + 64 + 16 * q, v);
                scale_i64(e, col + 64 + 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const long long x1 = pre_relu ? relu(x[i]) : x[i];
                    s[16 * q + i] = pass == 0 ? s[16 * q + i] + x1 : s[16 * q + i] - x1;
                }
            }
            fwht_fixed<64, 64>(s);
            if (post_relu) {
#pragma unroll
                for (int i = 0; i < 64; ++i) s[i] = relu(s[i]);
            }
            store_codes<64>(a, e.row, col + 64 * pass, s);
        } else {
            float s[64];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                int v[16];
                float x[16];
                load_acc16(e, col + 16 * q, v);
                scale_f32(e, col + 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) s[16 * q + i] = x[i];
                load_acc16(e, col + 64 + 16 * q, v);
                scale_f32(e, col + 64 + 16 * q, v, x);
#pragma unroll
                for (int i = 0; i < 16; ++i) s[16 * q + i] = pass == 0 ? s[16 * q + i] + x[i] : s[16 * q + i] - x[i];
            }
            fwht_fixed<64, 64>(s);
            if (post_relu || pre_relu) {
#pragma unroll
                for (int i = 0; i < 64; ++i) s[i] = relu(s[i]);
            }
            store_f32<64>(e.row, col + 64 * pass, s);
        }
    }
}

// ------------------------------------------------------------------ kernel

__global__ void __launch_bounds__(kThreads, 1)
    conv_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const ConvArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = a.stages;
    uint8_t *bar_area = smem + (size_t)S * a.stage_bytes;
    const uint32_t bar0 = smem_addr(bar_area);
    // barriers: full[S], conv[S], empty[S], acc_full, acc_empty, mma_done
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto conv_bar = [&](int s) { return bar0 + 8u * (S + s); };
    auto empty_bar = [&](int s) { return bar0 + 8u * (2 * S + s); };
    const uint32_t acc_full = bar0 + 8u * (3 * S);
    const uint32_t acc_empty = acc_full + 8;
    const uint32_t mma_done = acc_full + 16;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_area + 8 * (3 * S + 3));
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_area + 8 * (3 * S + 3) + 4);

    // A failure already recorded by this launch (or an earlier, unread one)
    // ends every CTA that has not started, so a fault cannot serialize waits.
    // One thread reads the word so the whole CTA takes the same decision.
    __shared__ int s_skip;
    if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int *>(a.err);
    __syncthreads();
    if (s_skip != 0) return;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    // tile coordinates
    const int tiles_per_img = a.tiles_w * a.tiles_h;
    const int img = blockIdx.x / tiles_per_img;
    const int rem = blockIdx.x - img * tiles_per_img;
    const int ty = rem / a.tiles_w;
    const int tx = rem - ty * a.tiles_w;
    const int ho0 = ty * a.th, wo0 = tx * a.tw;
    const int n0 = blockIdx.y * a.n_t;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(conv_bar(s), kConvThreads);
            mbar_init(empty_bar(s), 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(acc_empty, 128);
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_holder)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // per-tile bias codes, multipliers and dequant factors for the epilogue,
    // staged once (128-byte aligned, read with 16-byte vector loads)
    int *cb = reinterpret_cast<int *>(bar_area + a.const_off);
    for (int c = threadIdx.x; c < a.n_t; c += kThreads) {
        cb[c] = a.b_int[n0 + c];
        cb[256 + c] = a.mult[n0 + c];
        reinterpret_cast<float *>(cb)[512 + c] = a.deq[n0 + c];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;

    const int nchunks = (a.num_kb + a.chunk_kb - 1) / a.chunk_kb;

    if (warp == 0) {
        // ---------------------------------------------------------- TMA producer
        if (lane == 0) {
            const uint32_t tx_bytes = (uint32_t)(a.b_bytes + (a.gather ? 0 : a.raw_bytes));
            int issued_round[8];
            for (int s = 0; s < 8; ++s) issued_round[s] = -1;
            bool ok = true;
            for (int kb = 0; kb < a.num_kb && ok; ++kb) {
                const int s = kb % S, r = kb / S;
                if (!mbar_wait(empty_bar(s), (r & 1) ^ 1, abort_flag, a.err)) { ok = false; break; }
                const uint32_t st = smem_addr(smem + (size_t)s * a.stage_bytes);
                mbar_expect_tx(full_bar(s), tx_bytes);
                tma_load_2d(st + 16384, &tmB, full_bar(s), kb * kBlockK, n0);
                if (!a.gather) {
                    const int tap = kb / a.cin_kb;
                    const int c0 = (kb - tap * a.cin_kb) * kBlockK;
                    const int ky = tap / a.kw, kx = tap - (tap / a.kw) * a.kw;
                    tma_load_4d(st + 16384 + a.b_bytes, &tmA, full_bar(s), c0, wo0 * a.stride + kx - a.pad,
                                ho0 * a.stride + ky - a.pad, img);
                }
                issued_round[s] = r;
            }
            if (!ok) {
                // let our own copies land before the CTA unwinds
                for (int s = 0; s < S && s < 8; ++s)
                    if (issued_round[s] >= 0) {
                        const long long t0 = clock64();
                        while (!mbar_try_wait(full_bar(s), issued_round[s] & 1) && clock64() - t0 < kWaitLimitCycles) {
                        }
                    }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16(a.n_t);
            bool ok = true;
            for (int kb = 0; kb < a.num_kb && ok; ++kb) {
                const int s = kb % S, r = kb / S;
                const int ck = kb % a.chunk_kb;
                if (ck == 0 && kb > 0) {
                    const int ch = kb / a.chunk_kb;    // wait until chunk ch-1 was drained
                    if (!mbar_wait(acc_empty, (ch - 1) & 1, abort_flag, a.err)) { ok = false; break; }
                    tc_fence_after();
                }
                if (!mbar_wait(full_bar(s), r & 1, abort_flag, a.err)) { ok = false; break; }
                if (!mbar_wait(conv_bar(s), r & 1, abort_flag, a.err)) { ok = false; break; }
                tc_fence_after();
                const uint32_t st = smem_addr(smem + (size_t)s * a.stage_bytes);
                const uint64_t da = sdesc_sw128(st);
                const uint64_t db = sdesc_sw128(st + 16384);
#pragma unroll
                for (int kk = 0; kk < kBlockK / 16; ++kk)   // K = 16 per instruction, 32 bytes apart
                    umma_f16(tmem, da + (uint64_t)(2 * kk), db + (uint64_t)(2 * kk), idesc, (ck > 0 || kk > 0) ? 1u : 0u);
                umma_commit(empty_bar(s));
                if (ck == a.chunk_kb - 1 || kb == a.num_kb - 1) umma_commit(acc_full);
            }
            umma_commit(mma_done);
            const long long t0 = clock64();
            while (!mbar_try_wait(mma_done, 0) && clock64() - t0 < kWaitLimitCycles) {
            }
        }
    } else if (warp < 4) {
        // ---------------------------------------------------------- converters
        constexpr int kPasses = 512 / kConvThreads;   // 128 rows x 4 quarters per 64-wide block
        const int ct = threadIdx.x - 64;              // 0..kConvThreads-1
        if (!a.gather) {
            for (int kb = 0; kb < a.num_kb; ++kb) {
                const int s = kb % S, r = kb / S;
                if (!mbar_wait(full_bar(s), r & 1, abort_flag, a.err)) break;
                uint8_t *st = smem + (size_t)s * a.stage_bytes;
                const uint8_t *raw = st + 16384 + a.b_bytes;
                int4 v[kPasses];                       // all loads first, then convert and store
#pragma unroll
                for (int p = 0; p < kPasses; ++p) {
                    const int idx = p * kConvThreads + ct;
                    v[p] = *reinterpret_cast<const int4 *>(raw + (idx >> 2) * 64 + (idx & 3) * 16);
                }
#pragma unroll
                for (int p = 0; p < kPasses; ++p) {
                    const int idx = p * kConvThreads + ct;
                    const int m = idx >> 2, q = idx & 3;    // row, 16-element quarter of the 64-wide block
                    uint32_t h[8];
                    i8x4_to_f16x4((uint32_t)v[p].x, h[0], h[1]);
                    i8x4_to_f16x4((uint32_t)v[p].y, h[2], h[3]);
                    i8x4_to_f16x4((uint32_t)v[p].z, h[4], h[5]);
                    i8x4_to_f16x4((uint32_t)v[p].w, h[6], h[7]);
                    *reinterpret_cast<int4 *>(st + sw128_offset(m, 2 * q)) = make_int4((int)h[0], (int)h[1], (int)h[2], (int)h[3]);
                    *reinterpret_cast<int4 *>(st + sw128_offset(m, 2 * q + 1)) = make_int4((int)h[4], (int)h[5], (int)h[6], (int)h[7]);
                }
                fence_proxy_async_smem();
                mbar_arrive(conv_bar(s));
            }
        } else {
            // Small-channel layer: the tile's input window ((th-1)s+kh rows of
            // (tw-1)s+kw pixels, zero outside the image) is copied to shared
            // memory with coalesced byte loads, then the packed reduction index
            // k = (ky, kx, ci) is gathered from it through a per-CTA offset table.
            int *tab = reinterpret_cast<int *>(bar_area + 8 * (3 * S + 3) + 16);
            uint8_t *win = bar_area + a.win_off;
            const int taps = a.kh * a.kw;
            for (int k = ct; k < a.num_kb * kBlockK; k += kConvThreads) {
                const int tap = k / a.c, ci = k - tap * a.c;
                const int ky = tap / a.kw, kx = tap - ky * a.kw;
                tab[k] = tap < taps ? (ky * a.win_w + kx) * a.c + ci : -1;
            }
            {
                const int ix_lo = wo0 * a.stride - a.pad;
                const int row_b = a.win_w * a.c;
                const int b_lo = max(0, -ix_lo) * a.c, b_hi = min(a.win_w, a.w - ix_lo) * a.c;
                for (int r = 0; r < a.win_h; ++r) {
                    const int iy = ho0 * a.stride - a.pad + r;
                    const bool row_in = iy >= 0 && iy < a.h;
                    const int8_t *src = a.x + (((long long)img * a.h + (row_in ? iy : 0)) * a.w + ix_lo) * a.c;
                    for (int b = ct; b < row_b; b += kConvThreads)
                        win[r * row_b + b] = (row_in && b >= b_lo && b < b_hi) ? (uint8_t)__ldg(src + b) : (uint8_t)0;
                }
            }
            asm volatile("bar.sync 1, %0;" ::"r"(kConvThreads) : "memory");
            int rb[kPasses];
#pragma unroll
            for (int p = 0; p < kPasses; ++p) {
                const int m = (p * kConvThreads + ct) >> 2;
                rb[p] = ((m / a.tw) * a.stride * a.win_w + (m % a.tw) * a.stride) * a.c;
            }
            for (int kb = 0; kb < a.num_kb; ++kb) {
                const int s = kb % S, r = kb / S;
                if (!mbar_wait(full_bar(s), r & 1, abort_flag, a.err)) break;
                uint8_t *st = smem + (size_t)s * a.stage_bytes;
#pragma unroll
                for (int p = 0; p < kPasses; ++p) {
                    const int idx = p * kConvThreads + ct;
                    const int m = idx >> 2, q = idx & 3;
                    uint32_t w4[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int off = tab[kb * kBlockK + q * 16 + j];
                        const uint32_t b = off >= 0 ? (uint32_t)win[rb[p] + off] : 0u;
                        w4[j >> 2] |= b << (8 * (j & 3));
                    }
                    uint32_t h[8];
#pragma unroll
                    for (int j = 0; j < 4; ++j) i8x4_to_f16x4(w4[j], h[2 * j], h[2 * j + 1]);
                    *reinterpret_cast<int4 *>(st + sw128_offset(m, 2 * q)) = make_int4((int)h[0], (int)h[1], (int)h[2], (int)h[3]);
                    *reinterpret_cast<int4 *>(st + sw128_offset(m, 2 * q + 1)) = make_int4((int)h[4], (int)h[5], (int)h[6], (int)h[7]);
                }
                fence_proxy_async_smem();
                mbar_arrive(conv_bar(s));
            }
        }
    } else {
        // ---------------------------------------------------------- drains (chunk sums -> int32 partial)
        const uint32_t t_acc = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const uint32_t t_part = t_acc + (uint32_t)a.part_col;
        for (int ch = 0; ch + 1 < nchunks; ++ch) {
            if (!mbar_wait(acc_full, ch & 1, abort_flag, a.err)) break;
            tc_fence_after();
            for (int col = 0; col < a.n_t; col += 32) {
                uint32_t r[32];
                tmem_ld32(t_acc + col, r);
                if (ch > 0) {
                    uint32_t p[32];
                    tmem_ld32(t_part + col, p);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = (uint32_t)(__float2int_rn(__uint_as_float(r[i])) + (int)p[i]);
                } else {
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = (uint32_t)__float2int_rn(__uint_as_float(r[i]));
                }
                tmem_st32(t_part + col, r);
            }
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(acc_empty);
        }
    }

    // -------------------------------------------------------------- final epilogue, all eight warps
    // Warps w and w+4 share TMEM lane quadrant w%4 and split the column groups.
    // mma_done completes exactly once, after the last MMA (and hence after the
    // last drain, which the MMA issuer waited for).
    __syncwarp();
    bool fin = mbar_wait(mma_done, 0, abort_flag, a.err);
    fin = __all_sync(0xffffffffu, fin);
    tc_fence_after();
    const int esz = a.out_f32 ? 4 : 1;
    const int row_bytes = a.n_t * esz, row_stride = row_bytes + 16;
    if (fin) {
        const int quad = warp & 3;
        const int row = quad * 32 + lane;
        EpiCtx e;
        e.b_int = cb;
        e.mult = cb + 256;
        e.deq = reinterpret_cast<const float *>(cb + 512);
        e.t_acc = tmem + ((uint32_t)(quad * 32) << 16);
        e.t_part = e.t_acc + (uint32_t)a.part_col;
        e.has_part = nchunks > 1;
        // output tile staged in the (now idle) pipeline buffers, rows padded by
        // 16 bytes so 8 consecutive rows fall in 8 different bank groups
        e.row = smem + (size_t)row * row_stride;
        const int G = max(32, max(a.hb_out, a.hb_next));
        const int mine = warp >> 2;                // warps 4-7 take even groups, 0-3 odd
        int gi = 0;
        for (int col = 0; col < a.n_t; col += G, ++gi) {
            if ((gi & 1) != (mine ^ 1)) continue;
            if (G == 32) epi_group<32>(e, a, col);
            else if (G == 64) epi_group<64>(e, a, col);
            else epi_group128(e, a, col);
        }
    }
    __syncthreads();
    if (*abort_flag == 0) {
        // coalesced copy-out: consecutive threads write consecutive 16-byte chunks
        const int cpr = row_bytes >> 4;
        for (int j = threadIdx.x; j < kTileM * cpr; j += kThreads) {
            const int r = j / cpr, c = j - r * cpr;
            const int oy = ho0 + r / a.tw, ox = wo0 + r % a.tw;
            if (oy < a.ho && ox < a.wo) {
                const long long pix = ((long long)img * a.ho + oy) * a.wo + ox;
                const int4 v = *reinterpret_cast<const int4 *>(smem + (size_t)r * row_stride + c * 16);
                *reinterpret_cast<int4 *>(static_cast<uint8_t *>(a.y) + (pix * a.co + n0) * esz + c * 16) = v;
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

}  // namespace

cudaError_t launch_conv(const CUtensorMap &tmA, const CUtensorMap &tmB, const ConvArgs &a, int smem_bytes, cudaStream_t s) {
    static int configured_smem = 0;
    if (smem_bytes > configured_smem) {
        cudaError_t e = cudaFuncSetAttribute(conv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return e;
        configured_smem = smem_bytes;
    }
    dim3 grid((unsigned)(a.n * a.tiles_w * a.tiles_h), (unsigned)(a.co / a.n_t));
    conv_kernel<<<grid, kThreads, smem_bytes, s>>>(tmA, tmB, a);
    return cudaGetLastError();
}

}  // namespace hatq
