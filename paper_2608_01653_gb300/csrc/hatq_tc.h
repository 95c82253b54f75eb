// Device helpers shared by the tensor-core kernels: mbarrier waits with a
// cycle limit, TMA tile loads, tcgen05 descriptors / MMA / tensor-memory
// loads and stores, and the exact integer requantization and Sylvester
// butterflies of the epilogues. Every wait that can spin is bounded.
#pragma once

#include <cuda.h>
#include <cstdint>

#include "hatq_internal.h"

namespace hatq {
namespace tc {

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
// another role raised the abort flag, or the device error word is set).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag, int *err,
                                          long long limit = kWaitLimitCycles) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t spin = 1;; ++spin) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((spin & 63) == 0) {
            if (*abort_flag) return false;
            if (*reinterpret_cast<volatile int *>(err) != 0) { *abort_flag = 1; return false; }
            if (clock64() - t0 > limit) {
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
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *tm, uint32_t bar, int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(tm), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
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

// D (+)= A * B^T with the A operand in TMEM (lane = row, two fp16 per 32-bit
// column, K ascending) and B described in shared memory.
__device__ __forceinline__ void umma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// D (+)= A * B^T with both operands described in shared memory.
__device__ __forceinline__ void umma_f16_ss(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
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

// The same rounding for 33 <= n <= 62 on the 32-bit halves of v (s = n - 32,
// kh = 2^(s-1) - 1): v + 2^(n-1) - 1 + bit_n(v) has the high word
// hi + kh + c, where c is the carry out of the low word, lo + (2^32 - 1) + bit,
// i.e. c = [lo or bit nonzero]; its shift by n is that high word shifted by s.
__device__ __forceinline__ int requant8_hi(long long v, int s, int kh) {
    const uint32_t lo = (uint32_t)v;
    const int hi = (int)((unsigned long long)v >> 32);
    const uint32_t bit = (uint32_t)(hi >> s) & 1u;
    const int c = (int)min(lo | bit, 1u);
    return min(max((hi + kh + c) >> s, -127), 127);
}
// n = 32: v + 2^31 - 1 + bit_32(v) carries out of the low word iff lo + bit > 2^31.
__device__ __forceinline__ int requant8_32(long long v) {
    const uint32_t lo = (uint32_t)v;
    const int hi = (int)((unsigned long long)v >> 32);
    const int c = (lo > 0x80000000u || (lo == 0x80000000u && (hi & 1))) ? 1 : 0;
    return min(max(hi + c, -127), 127);
}
// The same rounding for 32 <= n <= 62 with only the lower clamp (the
// saturating pack below does the upper one): the 64-bit sum
// v + (2^(n-1) - 1) + bit_n(v) (kadd = 2^(n-1) - 1, s = n - 32; no overflow for
// |v| < 2^62) shifted by n is its high word shifted by s.
__device__ __forceinline__ int requant8_lo(long long v, long long kadd, int s) {
    const int bit = ((int)((unsigned long long)v >> 32) >> s) & 1;
    const unsigned long long u = (unsigned long long)(v + kadd) + (unsigned long long)bit;
    return max((int)(u >> 32) >> s, -127);
}
// bytes (q0, q1, q2, q3) of a word, each q saturated to [-128, 127]
__device__ __forceinline__ uint32_t pack4_sat(int q0, int q1, int q2, int q3) {
    uint32_t hi, d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(hi) : "r"(q3), "r"(q2), "r"(0u));
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(hi));
    return d;
}
// requant8 with the 32-bit-piece paths for shifts >= 32 (n is uniform).
__device__ __forceinline__ int requant8_any(long long v, int n) {
    if (n > 32) return requant8_hi(v, n - 32, (1 << (n - 33)) - 1);
    return n == 32 ? requant8_32(v) : requant8(v, n);
}

// Low bytes of four codes in [-127, 127] packed into one word.
__device__ __forceinline__ uint32_t pack4(int q0, int q1, int q2, int q3) {
    return __byte_perm(__byte_perm((uint32_t)q0, (uint32_t)q1, 0x0040), __byte_perm((uint32_t)q2, (uint32_t)q3, 0x0040),
                       0x5410);
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

}  // namespace tc
}  // namespace hatq
