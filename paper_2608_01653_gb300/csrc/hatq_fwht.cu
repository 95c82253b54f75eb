// Online activation transform + INT8 quantization (the activation side of
// HaTQ's double-Hadamard operator, Eq. double_hadamard_quantization, with the
// butterfly evaluation of the Sylvester transform, Eq. supp_sylvester, and
// the normalization folded into the quantization scale, as the deployment
// realization of the supplementary material describes).
//
// Memory-bound: every element is read once and written once. A warp owns a
// contiguous 512-element span of the flattened NHWC tensor (16 elements per
// lane, one 16-byte load for INT8, two for FP16), so any Hadamard block
// (hb <= 256, hb | C, 16 | C) lies inside one warp: the first log2(min(hb,16))
// butterfly stages run inside a lane, the rest across lanes with __shfl_xor.
//
// INT8 entry: the integer butterfly runs on sign-extended int32 elements
// (cross-lane stages as one shuffle and one multiply-add by +-1), then
// y = clamp(round_half_even(M_q v / 2^n_q)), for n_q >= 32 in 32-bit pieces.
// FP16 entry: fp32 butterfly, y = clamp(rint(v * inv)), inv = 1/(sqrt(hb) s).
#include <cuda_fp16.h>

#include "hatq_internal.h"

namespace hatq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// 16 int8 codes -> 16 sign-extended int32 (prmt selector bit 3 replicates the sign).
__device__ __forceinline__ void unpack_i8x16_i32(const int4 raw, int (&v)[16]) {
    const uint32_t w[4] = {(uint32_t)raw.x, (uint32_t)raw.y, (uint32_t)raw.z, (uint32_t)raw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        v[4 * i + 0] = (int)prmt(w[i], 0u, 0x8880u);
        v[4 * i + 1] = (int)prmt(w[i], 0u, 0x9991u);
        v[4 * i + 2] = (int)prmt(w[i], 0u, 0xAAA2u);
        v[4 * i + 3] = (int)prmt(w[i], 0u, 0xBBB3u);
    }
}

// Sylvester butterfly over the 16 elements of one lane plus the cross-lane
// stages; afterwards each element holds (H~_hb x)_j. In a cross-lane stage
// the upper lane of a pair keeps partner - own, the lower own + partner.
__device__ __forceinline__ void butterfly_i32(int (&v)[16], int hb, int lane) {
#pragma unroll
    for (int h = 1; h < 16; h <<= 1) {
        if (h >= hb) break;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            if (i & h) continue;
            const int a = v[i], b = v[i + h];
            v[i] = a + b;
            v[i + h] = a - b;
        }
    }
#pragma unroll
    for (int m = 1; m < 16; m <<= 1) {
        if (16 * m >= hb) break;
        const int sgn = (lane & m) ? -1 : 1;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int p = __shfl_xor_sync(0xffffffffu, v[i], m);
            v[i] = p + sgn * v[i];
        }
    }
}

__device__ __forceinline__ void butterfly_f32(float (&f)[16], int hb, int lane) {
#pragma unroll
    for (int h = 1; h < 16; h <<= 1) {
        if (h >= hb) break;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            if (i & h) continue;
            const float a = f[i], b = f[i + h];
            f[i] = a + b;
            f[i + h] = a - b;
        }
    }
#pragma unroll
    for (int m = 1; m < 16; m <<= 1) {
        if (16 * m >= hb) break;
        const bool upper = (lane & m) != 0;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float p = __shfl_xor_sync(0xffffffffu, f[i], m);
            f[i] = upper ? p - f[i] : f[i] + p;
        }
    }
}

// round(P / 2^n) half to even, clamped to [-127, 127].
__device__ __forceinline__ int requant(long long P, int n) {
    long long q = P;
    if (n > 0) q = (P + ((1LL << (n - 1)) - 1) + ((P >> n) & 1)) >> n;
    q = q < -127 ? -127 : (q > 127 ? 127 : q);
    return (int)q;
}

__device__ __forceinline__ int clamp127(int v) { return v < -127 ? -127 : (v > 127 ? 127 : v); }

// requant for 32 <= n <= 62 with k = 2^(n-1) - 1 and s = n - 32: P + k + bit_n(P)
// stays below 2^63 (|P| < 2^62) and its arithmetic shift by n is the high word
// shifted by s.
__device__ __forceinline__ int requant_hi(long long P, int s, long long k) {
    const uint32_t bit = ((uint32_t)((unsigned long long)P >> 32) >> s) & 1u;
    const long long u = P + k + (long long)bit;
    return clamp127((int)(u >> 32) >> s);
}
// round(P / 2^n) half to even for 1 <= n <= 30 in 32-bit arithmetic (the
// multiplier rule keeps |P| < 2^30, so P + 2^(n-1) does not overflow), clamped.
__device__ __forceinline__ int requant32(int P, int n, int k) {
    return clamp127((P + k + ((P >> n) & 1)) >> n);
}
__device__ __forceinline__ uint32_t pack4p(int a, int b, int c, int d) {
    return __byte_perm(__byte_perm((uint32_t)a, (uint32_t)b, 0x0040), __byte_perm((uint32_t)c, (uint32_t)d, 0x0040), 0x5410);
}


// MODE 0: static scale. MODE 1: scale from the dynamic parameter block.
// MODE 2: max-abs pass of the dynamic mode (no store).
template <bool F16, int MODE>
__global__ void __launch_bounds__(kThreads) act_quant_kernel(ActQuantArgs a) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * kThreads + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * kThreads) >> 5;
    const long long tiles = (a.total + 511) >> 9;
    long long mult = a.mult;
    int shift = a.shift;
    float inv = a.inv;
    if (MODE == 1 && !F16 && a.dyn->packed) return;   // the packed-pair pass quantizes this tensor
    if (MODE == 1) {
        mult = a.dyn->mult;
        shift = a.dyn->shift;
        inv = a.dyn->inv;
    }
    uint32_t local_max = 0;
    float local_maxf = 0.f;
    // Software pipelining: the loads of this warp's next two tiles are in
    // flight while the current tile is transformed and stored.
    int4 cur0 = make_int4(0, 0, 0, 0), cur1 = make_int4(0, 0, 0, 0);
    int4 mid0 = make_int4(0, 0, 0, 0), mid1 = make_int4(0, 0, 0, 0);
    auto load_tile = [&](long long t, int4 &v0, int4 &v1) {
        const long long e0 = (t << 9) + lane * 16;
        v0 = make_int4(0, 0, 0, 0);
        v1 = make_int4(0, 0, 0, 0);
        if (t < tiles && e0 < a.total) {
            if (!F16) {
                v0 = __ldg(reinterpret_cast<const int4 *>(static_cast<const int8_t *>(a.x) + e0));
            } else {
                const int4 *p = reinterpret_cast<const int4 *>(static_cast<const __half *>(a.x) + e0);
                v0 = __ldg(p);
                v1 = __ldg(p + 1);
            }
        }
    };
    load_tile(warp, cur0, cur1);
    load_tile(warp + nwarps, mid0, mid1);
    for (long long t = warp; t < tiles; t += nwarps) {
        int4 nxt0, nxt1;
        load_tile(t + 2 * nwarps, nxt0, nxt1);
        const long long e0 = (t << 9) + lane * 16;
        const bool valid = e0 < a.total;
        if (!F16) {
            int v[16];
            unpack_i8x16_i32(cur0, v);
            butterfly_i32(v, a.hb, lane);
            if (MODE == 2) {
#pragma unroll
                for (int k = 0; k < 16; ++k) local_max = max(local_max, (uint32_t)abs(v[k]));
            } else if (valid) {
                uint32_t o[4];
                const int m32 = (int)mult;            // M_q < 2^31
                if (shift >= 1 && shift <= 30) {
                    // M_q 127 hb < 2^30: the products fit 32 bits
                    const int k = (1 << (shift - 1)) - 1;
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        o[i] = pack4p(requant32(m32 * v[4 * i], shift, k), requant32(m32 * v[4 * i + 1], shift, k),
                                      requant32(m32 * v[4 * i + 2], shift, k), requant32(m32 * v[4 * i + 3], shift, k));
                } else if (shift >= 32) {
                    const int sh = shift - 32;
                    const long long k = (1LL << (shift - 1)) - 1;
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        o[i] = pack4p(requant_hi((long long)m32 * v[4 * i], sh, k), requant_hi((long long)m32 * v[4 * i + 1], sh, k),
                                      requant_hi((long long)m32 * v[4 * i + 2], sh, k), requant_hi((long long)m32 * v[4 * i + 3], sh, k));
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        o[i] = pack4p(requant((long long)m32 * v[4 * i], shift), requant((long long)m32 * v[4 * i + 1], shift),
                                      requant((long long)m32 * v[4 * i + 2], shift), requant((long long)m32 * v[4 * i + 3], shift));
                }
                *reinterpret_cast<int4 *>(a.y + e0) = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
            }
        } else {
            float f[16];
            const uint32_t w[8] = {(uint32_t)cur0.x, (uint32_t)cur0.y, (uint32_t)cur0.z, (uint32_t)cur0.w,
                                   (uint32_t)cur1.x, (uint32_t)cur1.y, (uint32_t)cur1.z, (uint32_t)cur1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
                f[2 * i] = v.x;
                f[2 * i + 1] = v.y;
            }
            butterfly_f32(f, a.hb, lane);
            if (MODE == 2) {
#pragma unroll
                for (int i = 0; i < 16; ++i) local_maxf = fmaxf(local_maxf, fabsf(f[i]));
            } else if (valid) {
                // clamp(rint(f * inv)): clamping to [-127, 127] first and adding
                // 1.5 * 2^23 rounds half to even into the low mantissa bits, whose
                // low byte is the two's-complement code
                uint32_t q[16];
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    q[i] = __float_as_uint(fminf(fmaxf(f[i] * inv, -127.f), 127.f) + 12582912.f);
                uint32_t o[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) o[i] = pack4p((int)q[4 * i], (int)q[4 * i + 1], (int)q[4 * i + 2], (int)q[4 * i + 3]);
                *reinterpret_cast<int4 *>(a.y + e0) = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
            }
        }
        cur0 = mid0;
        cur1 = mid1;
        mid0 = nxt0;
        mid1 = nxt1;
    }
    if (MODE == 2) {
        uint32_t m = F16 ? __float_as_uint(local_maxf) : local_max;   // nonnegative floats order as integers
        m = __reduce_max_sync(0xffffffffu, m);
        if (lane == 0 && m) atomicMax(&a.dyn->maxbits, m);
    }
}

// ------------------------------------------------------------------ dynamic affine (PTQ) activations
// Eqs. uniform_q, affine_q with the range extended to include zero:
// lo = min(min v, 0), hi = max(max v, 0), s = (hi - lo) / 255,
// z = clamp(round(-lo / s), 0, 255), x_int = clamp(round(v / s) + z, 0, 255);
// the layer consumes the centred codes x_int - z (int16, in [-255, 255]).
// v = T x is the fp32 butterfly of the FP16 input (T the normalized block
// transform of a DH layer; the identity for hb = 1).

// order-preserving unsigned key of a float (larger float, larger key)
__device__ __forceinline__ unsigned int float_key(float f) {
    const unsigned int b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_float(unsigned int k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// MODE 0: range pass (max v, max -v). MODE 1: quantize to centred int16 codes.
template <int MODE>
__global__ void __launch_bounds__(kThreads) act_affine_kernel(AffineQuantArgs a) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * kThreads + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * kThreads) >> 5;
    const long long tiles = (a.total + 511) >> 9;
    const float norm = 1.0f / sqrtf((float)a.hb);     // exact for the power-of-four blocks
    float vmax = -3.0e38f, vmin = 3.0e38f;
    float inv_s = 0.f, z = 0.f;
    if (MODE == 1) {
        inv_s = a.p->inv_s;
        z = a.p->z;
    }
    for (long long t = warp; t < tiles; t += nwarps) {
        const long long e0 = (t << 9) + lane * 16;
        const bool valid = e0 < a.total;
        int4 v0 = make_int4(0, 0, 0, 0), v1 = make_int4(0, 0, 0, 0);
        if (valid) {
            const int4 *p = reinterpret_cast<const int4 *>(static_cast<const __half *>(a.x) + e0);
            v0 = __ldg(p);
            v1 = __ldg(p + 1);
        }
        float f[16];
        const uint32_t w[8] = {(uint32_t)v0.x, (uint32_t)v0.y, (uint32_t)v0.z, (uint32_t)v0.w,
                               (uint32_t)v1.x, (uint32_t)v1.y, (uint32_t)v1.z, (uint32_t)v1.w};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
            f[2 * i] = v.x;
            f[2 * i + 1] = v.y;
        }
        butterfly_f32(f, a.hb, lane);
#pragma unroll
        for (int i = 0; i < 16; ++i) f[i] *= norm;
        if (!valid) continue;
        if (MODE == 0) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                vmax = fmaxf(vmax, f[i]);
                vmin = fminf(vmin, f[i]);
            }
        } else {
            uint32_t o[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float q0 = fminf(fmaxf(rintf(f[2 * i] * inv_s) + z, 0.f), 255.f) - z;
                const float q1 = fminf(fmaxf(rintf(f[2 * i + 1] * inv_s) + z, 0.f), 255.f) - z;
                o[i] = ((uint32_t)(uint16_t)(int16_t)(int)q0) | ((uint32_t)(uint16_t)(int16_t)(int)q1 << 16);
            }
            int4 *dst = reinterpret_cast<int4 *>(a.y + e0);
            dst[0] = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
            dst[1] = make_int4((int)o[4], (int)o[5], (int)o[6], (int)o[7]);
        }
    }
    if (MODE == 0) {
        unsigned int kmax = float_key(vmax), kneg = float_key(-vmin);
        kmax = __reduce_max_sync(0xffffffffu, kmax);
        kneg = __reduce_max_sync(0xffffffffu, kneg);
        if (lane == 0) {
            atomicMax(&a.p->max_key, kmax);
            atomicMax(&a.p->negmin_key, kneg);
        }
    }
}

// s, z from the range (fp64 arithmetic on the fp32 extremes); a zero range gives (1, 0)
__global__ void act_affine_params_kernel(AffineParams *p, float *params_out) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const double hi = fmax((double)key_float(p->max_key), 0.0);
    const double lo = fmin(-(double)key_float(p->negmin_key), 0.0);
    double s = 1.0, z = 0.0;
    if (hi - lo > 0.0) {
        s = (hi - lo) / 255.0;
        z = fmin(fmax(rint(-lo / s), 0.0), 255.0);
    }
    p->s = (float)s;
    p->inv_s = (float)(1.0 / s);
    p->z = (float)z;
    if (params_out) {
        params_out[0] = (float)s;
        params_out[1] = (float)z;
    }
}

// INT8 entry, static scale, blocks of at most 64: a lane owns 64 consecutive
// elements (four 16-byte loads; the warp's loads cover 2 KB contiguously), so
// every butterfly stage runs inside the lane without shuffles. SMALL: the
// requantization fits 32-bit words (shift <= 30 under the multiplier rule).
template <int HB, bool SMALL>
__global__ void __launch_bounds__(kThreads) act_quant_i8_wide_kernel(ActQuantArgs a) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * kThreads + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * kThreads) >> 5;
    const long long tiles = (a.total + 2047) >> 11;
    const int m32 = (int)a.mult;
    const int shift = a.shift;
    const int k32 = shift >= 1 ? (1 << (shift - 1)) - 1 : 0;
    const int sh = shift - 32;
    const long long k64 = shift >= 1 ? (1LL << (shift - 1)) - 1 : 0;
    auto load = [&](long long t, int4 (&r)[4]) {
        const long long e0 = (t << 11) + lane * 64;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            r[q] = make_int4(0, 0, 0, 0);
            if (t < tiles && e0 + 16 * q < a.total)
                r[q] = __ldg(reinterpret_cast<const int4 *>(static_cast<const int8_t *>(a.x) + e0 + 16 * q));
        }
    };
    int4 cur[4], nxt[4];
    load(warp, cur);
    for (long long t = warp; t < tiles; t += nwarps) {
        load(t + nwarps, nxt);
        const long long e0 = (t << 11) + lane * 64;
        int v[64];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            int u[16];
            unpack_i8x16_i32(cur[q], u);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[16 * q + i] = u[i];
        }
#pragma unroll
        for (int h = 1; h < HB; h <<= 1) {
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                if (i & h) continue;
                const int x = v[i], y = v[i + h];
                v[i] = x + y;
                v[i + h] = x - y;
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (e0 + 16 * q >= a.total) break;
            uint32_t o[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                int c[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int x = v[16 * q + 4 * i + j];
                    if (SMALL) c[j] = shift ? requant32(m32 * x, shift, k32) : clamp127(m32 * x);
                    else c[j] = shift >= 32 ? requant_hi((long long)m32 * x, sh, k64) : requant((long long)m32 * x, shift);
                }
                o[i] = pack4p(c[0], c[1], c[2], c[3]);
            }
            *reinterpret_cast<int4 *>(a.y + e0 + 16 * q) = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) cur[q] = nxt[q];
    }
}

// Two 16-bit lanes per 32-bit word. A lane owns 128 consecutive elements and
// word j carries elements j (low half) and 64 + j (high half) as the integer
// lo + 65536 hi. Integer addition is linear, so one 32-bit add or subtract is
// a butterfly on both halves, and blocks of at most 64 never mix the halves.
// The bytes enter biased by 128 (v ^ 0x80); the first stage removes that bias
// and adds kBlo to the low half of every output, so at the end the low half
// is nonnegative and the word's bit pattern is the pair (lo, hi) of signed
// 16-bit values (|y| <= 127 * 64 < 2^15).
struct SwarParams {
    uint32_t clo;        // s16x2 lower clamp bound -vmax of y, plus the biases
    uint32_t clow, chigh; // requantization addends of the low and high halves
    uint32_t mult;
    int shift;
};

__device__ __forceinline__ uint32_t max_s16x2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.s16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}
// bytes (q0, q1, q2, q3) of a word, each q saturated to [-128, 127]
__device__ __forceinline__ uint32_t pack4s(int q0, int q1, int q2, int q3) {
    uint32_t hi, d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(hi) : "r"(q3), "r"(q2), "r"(0u));
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(hi));
    return d;
}

// TIES: rounding ties M y = 2^(n-1) (mod 2^n) can occur, so the half-to-even
// correction is applied; otherwise round half up is the same function.
template <int HB, bool TIES>
__device__ __forceinline__ int swar_requant(uint32_t a, uint32_t c, uint32_t m, int n) {
    const int p = (int)(m * a + c);                 // M y + 2^(n-1) (- 1 with TIES), exact mod 2^32
    if (TIES) return (p + ((p >> n) & 1)) >> n;
    return p >> n;
}

// Per-warp staging of the packed kernel: a 4 KB tile is 32 rows of 128 bytes,
// row l belonging to lane l; the 16-byte chunk q of row r sits at position
// q ^ (r & 7), so the coalesced copies (chunk 32 i + lane) and the row-wise
// reads and writes of a lane both touch 32 distinct banks per 8 lanes.
constexpr int kSwarWarps = 4;
constexpr int kSwarStages = 3;

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ int swz(int row, int chunk) { return row * 128 + ((chunk ^ (row & 7)) << 4); }

__device__ __forceinline__ uint32_t min_s16x2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("min.s16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// MODE 0: static scale, constants sp from the host. MODE 1: dynamic scale,
// constants from the parameter block (the kernel returns at once when the
// block says the packed pass does not apply; the general kernel then runs).
// MODE 2: the max-abs pass of the dynamic mode (max and min of the pairs, no
// stores).
template <int HB, bool TIES, int MODE>
__global__ void __launch_bounds__(kSwarWarps * 32) act_quant_i8_swar_kernel(ActQuantArgs a, SwarParams sp) {
    constexpr uint32_t kBlo = HB >= 2 ? 128u * HB : 0u;
    constexpr uint32_t kBias2 = 256u * 65537u;      // the two halves' input bias after one stage
    __shared__ __align__(128) uint8_t stage[kSwarWarps][kSwarStages][4096];
    if constexpr (MODE == 1) {
        const DynParams *dp = a.dyn;
        if (!dp->packed) return;
        sp.clo = dp->clo;
        sp.clow = dp->clow;
        sp.chigh = dp->chigh;
        sp.mult = (uint32_t)dp->mult;
        sp.shift = dp->shift;
    }
    uint32_t vmx = 0x80008000u, vmn = 0x7FFF7FFFu;  // running max / min of the (biased) pairs
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const long long warp = (long long)blockIdx.x * kSwarWarps + wib;
    const long long nwarps = (long long)gridDim.x * kSwarWarps;
    const long long tiles = (a.total + 4095) >> 12;
    const int8_t *xg = static_cast<const int8_t *>(a.x);
    // Copy tile t into a stage with zero fill past the end; one commit group
    // per call, empty when t is past the last tile.
    auto issue = [&](long long t, int slot) {
        if (t < tiles) {
            const long long e0 = t << 12;
            uint8_t *buf = stage[wib][slot];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int c = 32 * i + lane;
                const bool ok = e0 + 16 * c < a.total;
                const int8_t *src = ok ? xg + e0 + 16 * c : xg;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(buf + swz(c >> 3, c & 7))),
                             "l"(src), "r"(ok ? 16 : 0)
                             : "memory");
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int k = 0; k < kSwarStages; ++k) issue(warp + k * nwarps, k);
    int slot = 0;
    for (long long t = warp; t < tiles; t += nwarps) {
        asm volatile("cp.async.wait_group %0;" ::"n"(kSwarStages - 1) : "memory");
        __syncwarp();
        uint8_t *buf = stage[wib][slot];
        uint32_t x[64];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int4 ra = *reinterpret_cast<const int4 *>(buf + swz(lane, q));
            const int4 rb = *reinterpret_cast<const int4 *>(buf + swz(lane, q + 4));
            const uint32_t wa[4] = {(uint32_t)ra.x, (uint32_t)ra.y, (uint32_t)ra.z, (uint32_t)ra.w};
            const uint32_t wb[4] = {(uint32_t)rb.x, (uint32_t)rb.y, (uint32_t)rb.z, (uint32_t)rb.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t ae = (wa[i] ^ 0x80808080u) & 0x00FF00FFu, ao = (wa[i] ^ 0x80808080u) & 0xFF00FF00u;
                const uint32_t be = (wb[i] ^ 0x80808080u) & 0x00FF00FFu, bo = (wb[i] ^ 0x80808080u) & 0xFF00FF00u;
                const int j = 16 * q + 4 * i;
                x[j] = prmt(ae, be, 0x5410u);
                x[j + 1] = prmt(ao, bo, 0x4501u);
                x[j + 2] = prmt(ae, be, 0x7632u);
                x[j + 3] = prmt(ao, bo, 0x6723u);
            }
        }
        __syncwarp();                                  // the stage is free for this tile's codes
#pragma unroll
        for (int h = 1; h < HB; h <<= 1) {
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                if (i & h) continue;
                const uint32_t u = x[i], v = x[i + h];
                if (h == 1) {
                    // (u + v) carries the bias 2 * 128 of both halves, (u - v)
                    // none; kBlo on the first pair of a block is kBlo on its
                    // first input, which the transform spreads to every output
                    const uint32_t c = (i % HB) == 0 ? kBlo : 0u;
                    x[i] = u + v - kBias2 + c;
                    x[i + 1] = u - v + c;
                } else {
                    x[i] = u + v;
                    x[i + h] = u - v;
                }
            }
        }
        if constexpr (MODE == 2) {
            // zero-filled codes past the end transform to zeros, which do not change max |y|
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                vmx = max_s16x2(vmx, x[i]);
                vmn = min_s16x2(vmn, x[i]);
            }
        } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t oa[4], ob[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                int ql[4], qh[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    // y >= -vmax keeps the code >= -127; above, the saturating
                    // pack turns every code >= 128 into 127
                    const uint32_t w = max_s16x2(x[16 * q + 4 * i + k], sp.clo);
                    ql[k] = swar_requant<HB, TIES>(w & 0xFFFFu, sp.clow, sp.mult, sp.shift);
                    qh[k] = swar_requant<HB, TIES>((uint32_t)((int)w >> 16), sp.chigh, sp.mult, sp.shift);
                }
                oa[i] = pack4s(ql[0], ql[1], ql[2], ql[3]);
                ob[i] = pack4s(qh[0], qh[1], qh[2], qh[3]);
            }
            *reinterpret_cast<int4 *>(buf + swz(lane, q)) = make_int4((int)oa[0], (int)oa[1], (int)oa[2], (int)oa[3]);
            *reinterpret_cast<int4 *>(buf + swz(lane, q + 4)) = make_int4((int)ob[0], (int)ob[1], (int)ob[2], (int)ob[3]);
        }
        __syncwarp();
        const long long e0 = t << 12;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int c = 32 * i + lane;
            if (e0 + 16 * c < a.total)
                *reinterpret_cast<int4 *>(a.y + e0 + 16 * c) = *reinterpret_cast<const int4 *>(buf + swz(c >> 3, c & 7));
        }
        __syncwarp();                                  // every lane has read the stage back
        }
        issue(t + kSwarStages * nwarps, slot);
        slot = slot + 1 == kSwarStages ? 0 : slot + 1;
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if constexpr (MODE == 2) {
        // max |y| of the lane: low halves carry kBlo (HB >= 2) or 128 (HB = 1), high halves 0 or 128
        const int blo = HB >= 2 ? (int)kBlo : 128, bhi = HB >= 2 ? 0 : 128;
        int m = 0;
        if (vmx != 0x80008000u) {                      // the lane saw at least one tile
            const int lmx = (int)(int16_t)(vmx & 0xFFFFu) - blo, lmn = (int)(int16_t)(vmn & 0xFFFFu) - blo;
            const int hmx = ((int)vmx >> 16) - bhi, hmn = ((int)vmn >> 16) - bhi;
            m = max(max(abs(lmx), abs(lmn)), max(abs(hmx), abs(hmn)));
        }
        m = __reduce_max_sync(0xffffffffu, m);
        if (lane == 0 && m) atomicMax(&a.dyn->maxbits, (unsigned int)m);
    }
}

// FP16 entry, static scale, blocks of at most 64: a lane owns one 64-element
// block (128 bytes of fp16) of a 2048-element warp tile, staged in through
// shared memory like the packed INT8 pass (coalesced `cp.async` chunks, rows
// XOR-swizzled), transformed in fp32 in the lane and quantized as
// clamp(rint(f inv)); its 64 codes go back through the stage as half of a
// 128-byte row (chunk positions XOR-swizzled by row, conflict-free for 8
// lanes) and leave as coalesced 16-byte stores.
// MODE 0: static scale (a.inv). MODE 1: dynamic scale, inv from the parameter
// block. MODE 2: the max-abs pass of the dynamic mode (no stores).
template <int HB, int MODE>
__global__ void __launch_bounds__(kSwarWarps * 32) act_quant_f16_wide_kernel(ActQuantArgs a) {
    __shared__ __align__(128) uint8_t stage[kSwarWarps][kSwarStages][4096];
    float fmx = 0.f;
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const long long warp = (long long)blockIdx.x * kSwarWarps + wib;
    const long long nwarps = (long long)gridDim.x * kSwarWarps;
    const long long tiles = (a.total + 2047) >> 11;
    const uint8_t *xg = static_cast<const uint8_t *>(a.x);
    const float inv = MODE == 1 ? a.dyn->inv : a.inv;
    auto issue = [&](long long t, int slot) {
        if (t < tiles) {
            const long long e0 = t << 11;              // first element of the tile
            uint8_t *buf = stage[wib][slot];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int c = 32 * i + lane;           // 16-byte chunk = 8 elements
                const bool ok = e0 + 8 * c < a.total;
                const uint8_t *src = ok ? xg + 2 * (e0 + 8 * c) : xg;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(buf + swz(c >> 3, c & 7))),
                             "l"(src), "r"(ok ? 16 : 0)
                             : "memory");
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int k = 0; k < kSwarStages; ++k) issue(warp + k * nwarps, k);
    int slot = 0;
    for (long long t = warp; t < tiles; t += nwarps) {
        asm volatile("cp.async.wait_group %0;" ::"n"(kSwarStages - 1) : "memory");
        __syncwarp();
        uint8_t *buf = stage[wib][slot];
        float f[64];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const uint4 r = *reinterpret_cast<const uint4 *>(buf + swz(lane, q));
            const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
                f[8 * q + 2 * i] = v.x;
                f[8 * q + 2 * i + 1] = v.y;
            }
        }
        __syncwarp();                                  // the stage is free for this tile's codes
#pragma unroll
        for (int h = 1; h < HB; h <<= 1) {
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                if (i & h) continue;
                const float u = f[i], v = f[i + h];
                f[i] = u + v;
                f[i + h] = u - v;
            }
        }
        if constexpr (MODE == 2) {
            // zero-filled elements past the end transform to zeros
#pragma unroll
            for (int i = 0; i < 64; ++i) fmx = fmaxf(fmx, fabsf(f[i]));
            issue(t + kSwarStages * nwarps, slot);
            slot = slot + 1 == kSwarStages ? 0 : slot + 1;
            continue;
        } else {
        // clamp(rint(f inv)) as in the general kernel: the clamp first, then
        // 1.5 * 2^23 rounds half to even into the low mantissa byte
        const int orow = lane >> 1, ocol = 4 * (lane & 1);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t o[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint32_t c[4];
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    c[k] = __float_as_uint(fminf(fmaxf(f[16 * q + 4 * i + k] * inv, -127.f), 127.f) + 12582912.f);
                o[i] = pack4p((int)c[0], (int)c[1], (int)c[2], (int)c[3]);
            }
            *reinterpret_cast<uint4 *>(buf + orow * 128 + (((ocol + q) ^ (orow & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
        __syncwarp();
        const long long o0 = t << 11;                  // first code of the tile
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int c = 32 * i + lane;
            const int row = c >> 3;
            if (o0 + 16 * c < a.total)
                *reinterpret_cast<uint4 *>(a.y + o0 + 16 * c) =
                    *reinterpret_cast<const uint4 *>(buf + row * 128 + (((c & 7) ^ (row & 7)) << 4));
        }
        __syncwarp();                                  // every lane has read the stage back
        issue(t + kSwarStages * nwarps, slot);
        slot = slot + 1 == kSwarStages ? 0 : slot + 1;
        }
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if constexpr (MODE == 2) {
        // nonnegative floats order as their bit patterns
        const unsigned int m = __reduce_max_sync(0xffffffffu, __float_as_uint(fmx));
        if (lane == 0 && m) atomicMax(&a.dyn->maxbits, m);
    }
}

// round(num / den) half to even for num, den > 0.
__device__ long long div_rne(unsigned long long num, unsigned long long den) {
    unsigned long long q = num / den, r = num % den;
    if (2 * r > den || (2 * r == den && (q & 1))) ++q;
    return (long long)q;
}

// Dynamic parameters from the max-abs: INT8 entry uses the exact rational
// rho = 127 / max|v| (the 1/sqrt(hb) and s_in cancel), M = round(rho 2^n) with
// the largest n such that M < 2^31 and M 127 hb < 2^30 (the requantizer's
// 32-bit product bound; at least 15 bits in M); the scan starts at n = 55
// (127 * 2^55 < 2^63), and every n > 39 fails M < 2^31 for the max
// |v| <= 127 * 256 of this operator, so the result equals a scan from 62.
__global__ void act_dyn_params_kernel(DynParams *p, int f16, int hb, float s_in, float *s_used, int *err) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const unsigned int mb = p->maxbits;
    const double sq = sqrt((double)hb);
    if (mb == 0) {
        p->mult = 0; p->shift = 0; p->packed = 0;
        if (s_used) *s_used = 1.0f;
        return;
    }
    if (f16) {
        const float m = __uint_as_float(mb);
        p->inv = 127.0f / m;
        p->mult = 0; p->shift = 0;
        if (s_used) *s_used = (float)((double)m / (sq * 127.0));
        return;
    }
    int found = -1;
    long long M = 0;
    for (int n = 55; n >= 0; --n) {
        const long long m = div_rne(127ull << n, (unsigned long long)mb);
        if (m >= (1LL << 31)) continue;
        const unsigned long long worst = (unsigned long long)m * 127ull * (unsigned long long)hb;
        if (worst >= (1ull << 30)) continue;        // the requantizer's 32-bit product bound
        found = n; M = m;
        break;
    }
    if (found < 0 || M < (1LL << 14)) {
        atomicExch(err, kErrBounds);
        found = 0; M = 0;
    }
    p->mult = M;
    p->shift = found;
    p->packed = 0;
    // the packed-pair pass (blocks <= 64, 32-bit requantization, codes that step
    // by at most one): clamp bound vmax = the largest y <= 127 hb whose code is
    // <= 127, round half to even in full (ties are not excluded here)
    if (hb <= 64 && found >= 1 && found <= 30 && M >= 1 && M <= (1LL << found)) {
        auto rne = [&](long long v) { return (v + ((1LL << (found - 1)) - 1) + ((v >> found) & 1)) >> found; };
        long long lo = 0, hi = 127LL * hb;
        if (rne(M * hi) > 127) {
            while (lo < hi) {
                const long long mid = (lo + hi + 1) / 2;
                if (rne(M * mid) <= 127) lo = mid;
                else hi = mid - 1;
            }
        }
        const uint32_t blo = hb >= 2 ? 128u * hb : 128u, bhi = hb >= 2 ? 0u : 128u;
        const long long clo_lo = -hi + (long long)blo, clo_hi = -hi + (long long)bhi;
        p->clo = (uint32_t)(clo_lo & 0xFFFF) | ((uint32_t)(clo_hi & 0xFFFF) << 16);
        const uint32_t half = (1u << (found - 1)) - 1u;
        p->clow = half - (uint32_t)M * blo;
        p->chigh = half - (uint32_t)M * bhi;
        p->packed = 1;
    }
    if (s_used) *s_used = (float)(((double)s_in * (double)mb) / (sq * 127.0));
}

int num_sms() {
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 148;
    }
    return sms;
}

// One wave: the blocks of kernel `k` that are resident at once (the grid-stride
// loop then gives every warp the same number of tiles).
template <typename K>
int grid_for(long long total, K k) {
    const long long tiles = (total + 511) / 512;
    const long long want = (tiles + 7) / 8;           // 8 warps per block
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kThreads, 0) != cudaSuccess || per_sm < 1) per_sm = 4;
    const long long cap = (long long)num_sms() * per_sm;
    return (int)(want < 1 ? 1 : (want < cap ? want : cap));
}

}  // namespace

template <int HB>
cudaError_t launch_wide(const ActQuantArgs &a, cudaStream_t s) {
    // grid_for counts 512-element warp tiles; a wide tile is 2048 elements
    if (a.shift <= 30) {
        auto k = act_quant_i8_wide_kernel<HB, true>;
        k<<<grid_for((a.total + 3) / 4, k), kThreads, 0, s>>>(a);
    } else {
        auto k = act_quant_i8_wide_kernel<HB, false>;
        k<<<grid_for((a.total + 3) / 4, k), kThreads, 0, s>>>(a);
    }
    return cudaGetLastError();
}

// round(M y / 2^n) half to even, 64-bit host arithmetic (the kernels' function).
long long host_rne(long long p, int n) {
    if (n <= 0) return p;
    return (p + ((1LL << (n - 1)) - 1) + ((p >> n) & 1)) >> n;
}

// One wave of the packed kernel: its resident blocks, at most one warp per 4096-code tile.
template <typename K>
int swar_grid(const ActQuantArgs &a, K k) {
    const long long want = ((a.total + 4095) / 4096 + kSwarWarps - 1) / kSwarWarps;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kSwarWarps * 32, 0) != cudaSuccess || per_sm < 1)
        per_sm = 4;
    const long long cap = (long long)num_sms() * per_sm;
    return (int)(want < 1 ? 1 : (want < cap ? want : cap));
}

template <int HB>
cudaError_t launch_swar(const ActQuantArgs &a, cudaStream_t s) {
    const long long m = a.mult;
    const int n = a.shift;
    // |y| <= vmax keeps round(M y / 2^n) within [-127, 127]; with M <= 2^n the
    // codes step by at most one, so clamping y below at -vmax gives code -127
    // exactly where the clamp of the code would (codes above 127 saturate in
    // the pack).
    long long lo = 0, hi = 127LL * HB;
    if (host_rne(m * hi, n) > 127) {
        while (lo < hi) {
            const long long mid = (lo + hi + 1) / 2;
            if (host_rne(m * mid, n) <= 127) lo = mid;
            else hi = mid - 1;
        }
    }
    const long long vmax = hi;
    // A tie M y = 2^(n-1) (mod 2^n) needs |y| >= 2^(n-1-t), t the trailing zeros of M.
    int t = 0;
    while (t < n && ((m >> t) & 1) == 0) ++t;
    const bool ties = t < n && (1LL << (n - 1 - t)) <= vmax;
    const uint32_t blo = HB >= 2 ? 128u * HB : 128u, bhi = HB >= 2 ? 0u : 128u;
    auto pair = [](long long lo16, long long hi16) {
        return (uint32_t)(lo16 & 0xFFFF) | ((uint32_t)(hi16 & 0xFFFF) << 16);
    };
    SwarParams sp;
    sp.clo = pair(-vmax + blo, -vmax + bhi);
    const uint32_t half = (1u << (n - 1)) - (ties ? 1u : 0u);
    sp.mult = (uint32_t)m;
    sp.clow = half - (uint32_t)m * blo;
    sp.chigh = half - (uint32_t)m * bhi;
    sp.shift = n;
    if (ties) {
        auto k = act_quant_i8_swar_kernel<HB, true, 0>;
        k<<<swar_grid(a, k), kSwarWarps * 32, 0, s>>>(a, sp);
    } else {
        auto k = act_quant_i8_swar_kernel<HB, false, 0>;
        k<<<swar_grid(a, k), kSwarWarps * 32, 0, s>>>(a, sp);
    }
    return cudaGetLastError();
}

template <int HB, int MODE>
cudaError_t launch_f16_wide(const ActQuantArgs &a, cudaStream_t s) {
    auto k = act_quant_f16_wide_kernel<HB, MODE>;
    // swar_grid counts 4096-element tiles; a tile here is 2048 elements
    ActQuantArgs g = a;
    g.total = 2 * a.total;
    k<<<swar_grid(g, k), kSwarWarps * 32, 0, s>>>(a);
    return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_f16_wide_hb(const ActQuantArgs &a, cudaStream_t s) {
    switch (a.hb) {
        case 1: return launch_f16_wide<1, MODE>(a, s);
        case 2: return launch_f16_wide<2, MODE>(a, s);
        case 4: return launch_f16_wide<4, MODE>(a, s);
        case 8: return launch_f16_wide<8, MODE>(a, s);
        case 16: return launch_f16_wide<16, MODE>(a, s);
        case 32: return launch_f16_wide<32, MODE>(a, s);
        default: return launch_f16_wide<64, MODE>(a, s);
    }
}

cudaError_t launch_act_quant(const ActQuantArgs &a, cudaStream_t s) {
    // packed pairs: INT8 entry, blocks of at most 64, 32-bit requantization
    // (1 <= n <= 30) and M <= 2^n (codes step by at most one)
    if (!a.f16 && a.hb <= 64 && a.shift >= 1 && a.shift <= 30 && a.mult <= (1LL << a.shift)) {
        switch (a.hb) {
            case 1: return launch_swar<1>(a, s);
            case 2: return launch_swar<2>(a, s);
            case 4: return launch_swar<4>(a, s);
            case 8: return launch_swar<8>(a, s);
            case 16: return launch_swar<16>(a, s);
            case 32: return launch_swar<32>(a, s);
            case 64: return launch_swar<64>(a, s);
            default: break;
        }
    }
    if (a.f16) {
        if (a.hb <= 64) return launch_f16_wide_hb<0>(a, s);
        act_quant_kernel<true, 0><<<grid_for(a.total, act_quant_kernel<true, 0>), kThreads, 0, s>>>(a);
        return cudaGetLastError();
    }
    switch (a.hb) {
        case 1: return launch_wide<1>(a, s);
        case 2: return launch_wide<2>(a, s);
        case 4: return launch_wide<4>(a, s);
        case 8: return launch_wide<8>(a, s);
        case 16: return launch_wide<16>(a, s);
        case 32: return launch_wide<32>(a, s);
        case 64: return launch_wide<64>(a, s);
        default:
            act_quant_kernel<false, 0><<<grid_for(a.total, act_quant_kernel<false, 0>), kThreads, 0, s>>>(a);
            return cudaGetLastError();
    }
}

cudaError_t launch_act_affine(const AffineQuantArgs &a, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(a.p, 0, sizeof(AffineParams), s);
    if (e != cudaSuccess) return e;
    act_affine_kernel<0><<<grid_for(a.total, act_affine_kernel<0>), kThreads, 0, s>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    act_affine_params_kernel<<<1, 32, 0, s>>>(a.p, a.params_out);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    act_affine_kernel<1><<<grid_for(a.total, act_affine_kernel<1>), kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

// Packed-pair max-abs pass (mode 2) or quantize pass (mode 1) of the dynamic mode.
template <int HB>
cudaError_t launch_swar_dyn(const ActQuantArgs &a, int mode, cudaStream_t s) {
    SwarParams sp{};
    if (mode == 2) {
        auto k = act_quant_i8_swar_kernel<HB, false, 2>;
        k<<<swar_grid(a, k), kSwarWarps * 32, 0, s>>>(a, sp);
    } else {
        auto k = act_quant_i8_swar_kernel<HB, true, 1>;
        k<<<swar_grid(a, k), kSwarWarps * 32, 0, s>>>(a, sp);
    }
    return cudaGetLastError();
}

cudaError_t launch_swar_dyn_hb(const ActQuantArgs &a, int mode, cudaStream_t s) {
    switch (a.hb) {
        case 1: return launch_swar_dyn<1>(a, mode, s);
        case 2: return launch_swar_dyn<2>(a, mode, s);
        case 4: return launch_swar_dyn<4>(a, mode, s);
        case 8: return launch_swar_dyn<8>(a, mode, s);
        case 16: return launch_swar_dyn<16>(a, mode, s);
        case 32: return launch_swar_dyn<32>(a, mode, s);
        default: return launch_swar_dyn<64>(a, mode, s);
    }
}

// Dynamic scale: max-abs pass, one-thread parameter kernel, quantize pass. The
// INT8 entry with blocks <= 64 takes the packed-pair kernels; its quantize pass
// launches the packed kernel and the general one, and the parameter block
// (written on the device) lets exactly one of them work.
cudaError_t launch_act_dynamic(const ActQuantArgs &a, float s_in, float *s_used, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(a.dyn, 0, sizeof(DynParams), s);
    if (e != cudaSuccess) return e;
    const bool packed = !a.f16 && a.hb <= 64;
    const bool wide16 = a.f16 && a.hb <= 64;
    if (wide16) { if ((e = launch_f16_wide_hb<2>(a, s)) != cudaSuccess) return e; }
    else if (a.f16) act_quant_kernel<true, 2><<<grid_for(a.total, act_quant_kernel<true, 2>), kThreads, 0, s>>>(a);
    else if (packed) { if ((e = launch_swar_dyn_hb(a, 2, s)) != cudaSuccess) return e; }
    else act_quant_kernel<false, 2><<<grid_for(a.total, act_quant_kernel<false, 2>), kThreads, 0, s>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    act_dyn_params_kernel<<<1, 32, 0, s>>>(a.dyn, a.f16, a.hb, s_in, s_used, a.err);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (wide16) return launch_f16_wide_hb<1>(a, s);
    if (a.f16) {
        act_quant_kernel<true, 1><<<grid_for(a.total, act_quant_kernel<true, 1>), kThreads, 0, s>>>(a);
        return cudaGetLastError();
    }
    if (packed && (e = launch_swar_dyn_hb(a, 1, s)) != cudaSuccess) return e;
    act_quant_kernel<false, 1><<<grid_for(a.total, act_quant_kernel<false, 1>), kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace hatq
