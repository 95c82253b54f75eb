// Internal interface between the host side of libhatq (hatq_api.cu) and the
// kernel translation units. Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hatq.h"

namespace hatq {

// Records `msg` as the calling thread's hatq_last_error() and returns st.
hatq_status report(hatq_status st, const char *msg);

// Error word codes written by kernels (read back by hatq_sync_status).
enum : int { kErrNone = 0, kErrWaitTimeout = 1, kErrBounds = 2 };

// ---------------------------------------------------------------- quantize
struct ActQuantArgs {
    const void *x;        // int8 or fp16 NHWC
    int8_t *y;
    long long total;      // elements, multiple of 16
    int hb;               // 1..256
    int f16;              // input is fp16
    long long mult;       // static INT8 entry: M_q
    int shift;            //                    n_q
    float inv;            // static FP16 entry: 1 / (sqrt(hb) s_out)
    // dynamic mode: device parameter block written by the parameter kernel
    struct DynParams *dyn;
    int *err;
};

// Device-side parameters of the dynamic-scale mode (lives in the caller's workspace).
struct DynParams {
    unsigned int maxbits;   // max |H~ x| (integer, or fp32 bits for FP16 entry)
    int shift;
    long long mult;
    union {
        float inv;          // FP16 entry: 127 / max|v|
        uint32_t packed;    // INT8 entry: 1 when the packed-pair quantize pass applies (M <= 2^n, n <= 30, hb <= 64)
    };
    uint32_t clo, clow, chigh;  // the packed-pair pass's constants (lower clamp, low / high requant addends)
};
static_assert(sizeof(DynParams) == 32, "the dynamic-mode workspace is 32 bytes");

// Device-side state of the dynamic affine quantizer (Eqs. uniform_q, affine_q;
// lives in the caller's workspace): order-preserving keys of max v and of
// -min v (both taken with atomicMax from zero), then the parameters.
struct AffineParams {
    unsigned int max_key, negmin_key;
    float s, inv_s;      // step and its reciprocal (fp32, for the quantize pass)
    float z;             // zero point, an integer in [0, 255]
    int pad_[3];
};

struct AffineQuantArgs {
    const void *x;        // fp16 NHWC
    int16_t *y;           // centred codes x_int - z, NHWC
    long long total;      // elements, multiple of 16
    int hb;               // block of the input-side transform (1: none)
    AffineParams *p;
    float *params_out;    // device [2]: s, z (float)
};
cudaError_t launch_act_affine(const AffineQuantArgs &a, cudaStream_t s);

// ---------------------------------------------------------------- profiling
struct ProfileArgs {
    const int8_t *x;       // NHWC codes, n images of per_image elements
    long long per_image;   // h * w * c, a multiple of 16
    int n, hb;
    int *maxima;           // [n][2]: max|x|, max|H~_hb x|
};
cudaError_t launch_profile(const ProfileArgs &a, uint8_t *expands, cudaStream_t s);

cudaError_t launch_act_quant(const ActQuantArgs &a, cudaStream_t s);
cudaError_t launch_wait_selftest(int *err, long long limit_cycles, cudaStream_t s);
cudaError_t launch_act_dynamic(const ActQuantArgs &a, float s_in, float *s_used, cudaStream_t s);

// ---------------------------------------------------------------- conv
struct ConvArgs {
    int n, h, w, c;
    int ho, wo, co;                  // output pixels this launch computes (a sub-convolution's own grid)
    int kh, kw, stride, pad_y, pad_x;   // input row / column of output (oy, ox), tap (ky, kx): oy s + ky - pad_y
    // where output pixel (oy, ox) goes: pixel (oy ostride + ooy, ox ostride + oox) of a [n][y_h][y_w][co]
    // tensor (transposed convolutions write one output parity class per launch); with d2s = r >= 2 the
    // channels are rearranged depth-to-space into a [n][y_h r][y_w r][co / r^2] tensor
    int y_h, y_w, ostride, ooy, oox, d2s;
    int tw, th, tiles_w, tiles_h;    // output tile: tw x th pixels (tw * th == 128, tw a power of two)
    int tw_log2;
    int n_t;                         // output channels per tile
    int num_kb;                      // 64-wide reduction blocks
    int cin_kb;                      // reduction blocks per kernel tap (tiled loader)
    int half;                        // tiled loader, c % 64 == 32: a block is two 32-channel boxes
    int cin_h;                       // half: 32-channel pieces per kernel tap
    int gather;                      // small-channel loader
    int seg;                         // small-channel loader: reduction entries per kernel row (kw * c, padded to 8)
    int chunk_kb;                    // reduction blocks per exact fp32 chunk
    int stages;
    int tmem_cols;                   // TMEM columns allocated (power of two)
    int a_col, a_slots;              // TMEM column of the fp16 A-operand ring and its slots (sub x 32 columns each)
    int nbuf, buf_cols;              // 2: epilogue warpgroups alternate tiles; 1: they split columns (drains); n_t
    int num_tiles, n_tiles_n;        // output tiles in the launch, N tiles per M tile
    int stage_bytes, b_bytes, raw_bytes;
    int sub;                         // 64-wide reduction blocks per pipeline stage (1 or 2)
    int b_off, raw_off;              // offsets of the weight and INT8 (64-byte swizzled) boxes inside a stage
    int staging_bytes, row_stride;   // shared-memory output tiles after the stages
    int const_off;                   // offsets from the barrier area: epilogue constants,
    int win_off, win_h, win_w;       // small-channel input window and its size
    int win_pitch;                   // bytes per window row
    int win_tma;                     // 1: the producer loads the window by TMA (two buffers, win_buf bytes apart)
    int win_buf, win_tma_bytes;      //    buffer stride and bytes of one window box
    const int8_t *x;
    const int32_t *b_int;
    const int32_t *mult;
    const float *deq;
    int shift, hb_out, hb_next, act, out_f32;   // act: 1 = ReLU folded into the single requantization
    void *y;
    int *err;
    // general transition (Sec. general nonlinearities): shift = n_out, mult = M_out,
    // then the table and the input-side pair (mult_in, shift_in)
    // dynamic affine activations (Eq. affine_q): the operand holds centred int16 codes (128-byte box
    // rows), the float epilogue takes s from *affine_s: t = (s s_w,c / gamma_out) a + beta_c with
    // beta_c = b_bar_c / gamma_out in `deq`
    int affine;
    float inv_gamma;
    const float *affine_s;
    const float *s_w;
    int general, shift_in;
    int a_f16;                       // operand codes as fp16 in the TMA tile: the MMA reads A from shared memory
    int out_f16;                     // codes written as fp16
    int lut_off;                     // offset of the table copy from the barrier area
    long long mult_in;
    int8_t lut[256];
};

// the convolution kernel for layers whose activation blocks arrive as two 32-channel boxes (a.half),
// with sub 64-wide blocks per pipeline stage (compiled in its own translation unit)
using ConvKernelFn = void (*)(const CUtensorMap, const CUtensorMap, const ConvArgs);
ConvKernelFn conv_pieces_kernel(int sub);
cudaError_t launch_conv(const CUtensorMap &tmA, const CUtensorMap &tmB, const ConvArgs &a,
                        int smem_bytes, cudaStream_t s);

// GDN / IGDN transition kernel (hatq_gdn.cu).
struct GdnArgs {
    const int8_t *z;                 // [pixels][c] preactivation codes (read through the tensor map)
    int8_t *y;                       // [pixels][c] next-layer codes
    long long pixels;
    int c, inverse, hb_next, t, shift_in;
    unsigned long long P;            // R^2 ~ P / 2^t
    float sr;                        // sqrt(P / 2^t) (estimate only)
    long long mult_in;               // M_in
    const int32_t *b_pool;           // [c] B_i
    int *err;
    int num_tiles, nz;               // 128-pixel tiles, z tile buffers (1 or 2)
    int z_off, u_off, b_off, lut_off, bar_off;  // shared-memory offsets from the 1024-aligned base
    int tmem_cols;
};

cudaError_t launch_gdn(const CUtensorMap &tmZ, const CUtensorMap &tmG, const GdnArgs &a, int smem_bytes,
                       cudaStream_t s);

}  // namespace hatq
