/*
 * hatq.h - C ABI of the Hadamard-domain INT8 convolution library (libhatq.so).
 *
 * The operator is HaTQ's layer in integer-only form ("Hadamard-Domain Model
 * Quantization for Learned Image Coding"): a convolution unfolded as the
 * linear operator Y = X W^T (Eq. linear_operator) whose operands are quantized
 * in a Hadamard basis, either double-Hadamard (DH: activations and weights
 * transformed along C_in, Eq. double_hadamard_quantization) or weight-only
 * (WH: weights transformed along C_out and the output basis restored after
 * accumulation, Eq. weight_only_hadamard_quantization), with INT8 codes,
 * int32 accumulation (Eq. integer_accumulation) and fixed-point
 * requantization (Eqs. integer_fixed_point_scale, integer_hadamard_transition).
 *
 * Conventions shared by every entry point
 *  - Layout: activations NHWC (C contiguous), weights OHWI, all C-contiguous.
 *  - Ownership: the caller allocates and owns every buffer; no entry point
 *    allocates device memory. Device pointers must be 16-byte aligned.
 *  - An empty batch (n == 0) is a valid no-op; its pointers may be NULL.
 *  - Streams: device work is enqueued on `stream` (a cudaStream_t; NULL is the
 *    legacy default stream) and is asynchronous unless stated otherwise.
 *  - Errors: argument, shape, alignment and overflow errors are returned
 *    before anything is launched; a CUDA launch error returns HATQ_ERR_CUDA.
 *    Kernels that wait on barriers wait a bounded time; an expired wait
 *    records an error word that hatq_sync_status() reports as
 *    HATQ_ERR_TIMEOUT. hatq_last_error() gives a message for the calling
 *    thread's last failure.
 *  - Codes are symmetric INT8 in [-127, 127] (Eq. symmetric_q with b = 8);
 *    round() is round-half-to-even everywhere.
 *  - Hadamard transforms are block-diagonal Sylvester transforms
 *    I_{C/hb} (x) H_hb along the channel axis (Eq. supp_sylvester), hb a power
 *    of two dividing the channel count; the unnormalized transform H~ uses
 *    only additions and subtractions, its 1/sqrt(hb) is folded into scales.
 */
#ifndef HATQ_H
#define HATQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *hatq_stream;   /* same type as cudaStream_t */

typedef enum {
    HATQ_OK = 0,
    HATQ_ERR_INVALID_ARG = 1,   /* bad pointer, shape, alignment or value */
    HATQ_ERR_UNSUPPORTED = 2,   /* valid by the paper but not implemented here */
    HATQ_ERR_OVERFLOW = 3,      /* int32 accumulator or int64 requant bound violated */
    HATQ_ERR_CUDA = 4,          /* a CUDA runtime/driver call failed */
    HATQ_ERR_TIMEOUT = 5        /* a bounded device-side wait expired */
} hatq_status;

/* DH, WH: Eqs. double_hadamard_quantization, weight_only_hadamard_quantization.
 * TRANSFORM: the activation-side transform of the paper's single order m(C)
 * as a bias-free 1x1 convolution (supplementary, deployment realization),
 * prepared only by hatq_prepare_order_transform. */
typedef enum { HATQ_DH = 0, HATQ_WH = 1, HATQ_TRANSFORM = 2 } hatq_form;
/* Activation between layers. NONE and RELU are positively homogeneous and
 * fold into the single requantization of Eq. integer_hadamard_transition;
 * SILU and GELU are not and take the two-step transition of Sec. general
 * nonlinearities (preactivation codes, integer table, input-side rescale),
 * prepared with hatq_prepare_weights_general. */
typedef enum { HATQ_ACT_NONE = 0, HATQ_ACT_RELU = 1, HATQ_ACT_SILU = 2, HATQ_ACT_GELU = 3 } hatq_act;

/* What a layer input holds (hatq_layer, hatq_quantize_act). */
typedef enum {
    HATQ_IN_OPERAND = 0,  /* INT8 codes already in this layer's operand basis and scale */
    HATQ_IN_I8 = 1,       /* INT8 codes in the original basis at scale s_in */
    HATQ_IN_F16 = 2       /* IEEE fp16 real values (FP16 entry) */
} hatq_input_kind;

/* One convolution (Eq. linear_operator with D = C_in Kh Kw). */
typedef struct {
    int c_in, c_out;      /* channels; c_out % 16 == 0 */
    int kh, kw;           /* kernel size */
    int stride, pad;      /* stride >= 1, symmetric zero padding */
    int form;             /* hatq_form, from the static profile mask (Eq. layerwise_hadamard_selection) */
    int hb_in;            /* DH: Hadamard block along c_in (2..256, power of two), or c_in itself for a
                             layer in the paper's single order (c_in = m, see hatq_prepare_weights_order);
                             0 for WH */
    int hb_out;           /* WH: Hadamard block along c_out (16..128); 0 for DH */
} hatq_conv_desc;

/*
 * A prepared layer (Sec. deployment realization: transformed weights are
 * input-independent and stored after offline transformation).
 * The caller sets the six device pointers (sizes from hatq_prepared_sizes)
 * before hatq_prepare_weights fills them; every other field is written by
 * the library. opaque[] holds the library's tensor-memory-access descriptor
 * of w_f16 and must not be modified.
 */
typedef struct {
    hatq_conv_desc d;
    int act;              /* hatq_act */
    int hb_next;          /* block of the next layer's DH transform applied in this epilogue, 0 = none */
    int out_f32;          /* 1: dequantized float32 output; 0: INT8 codes at s_y */
    int shift;            /* shared right shift n (Eq. integer_fixed_point_scale) */
    int k_pad;            /* packed reduction length = columns of w_i8 / w_f16 */
    int gather;           /* 1: small-channel layer (c_in % 16 != 0): kernel row ky holds the kw*c_in
                             entries (kx, c_in) padded with zero weights to a multiple of 8 */
    float s_x;            /* scale of the INT8 operand this layer consumes */
    float s_y;            /* scale of the INT8 codes it emits */
    int8_t *w_i8;         /* [c_out][k_pad] weight codes w_int, K order (kh, kw, c_in); gather == 0: c_in
                             padded to a multiple of 64 per tap, except c_in % 64 == 32 (taps unpadded,
                             the total padded to a multiple of 64); gather == 1: kw*c_in padded to 8 per row */
    uint16_t *w_f16;      /* [c_out][k_pad] the same codes as IEEE fp16 (exact), tensor-core operand */
    int32_t *b_int;       /* [c_out] bias codes, Eq. supp_bias_quantization */
    int32_t *mult;        /* [c_out] multipliers M_c, Eq. integer_fixed_point_scale */
    float *deq;           /* [c_out] s_x s_w,c / gamma_out (float32 output mode) */
    float *s_w;           /* [c_out] per-output-channel weight scales */
    uint64_t opaque[16];
    /* general transition (act SILU / GELU), written by hatq_prepare_weights_general;
     * then `mult` / `shift` hold M_out / n_out of Eq. supp_general_output_scale */
    float s_z;            /* preactivation scale */
    float s_u;            /* activation-output scale */
    int shift_in;         /* n_in of Eq. supp_general_input_scale */
    int in_affine;        /* 1: prepared by hatq_prepare_weights_affine (centred int16 operand, float output) */
    long long mult_in;    /* M_in of Eq. supp_general_input_scale */
    int8_t lut[256];      /* phi_int of Eq. supp_general_activation at z = -127..127 (index z + 127) */
    int in_f16;           /* 1: the INT8 operand arrives as IEEE fp16 values (exact), see hatq_set_operand_format */
    int out_f16;          /* 1: the INT8 codes are written as IEEE fp16 values (exact) */
} hatq_prepared;

/*
 * Storage format of a prepared layer's operand and output codes (the values
 * are the same INT8 codes either way; the paper has no counterpart: this only
 * changes how they sit in memory). in_f16: hatq_conv2d_i8 and hatq_layer
 * (x_kind HATQ_IN_OPERAND) read x as fp16 [n][h][w][c_in]; the tensor cores
 * then take the operand straight from the TMA tile in shared memory, with no
 * conversion per output-channel tile. out_f16: the layer writes its codes as
 * fp16 (twice the bytes), the operand format of a next layer with in_f16.
 * Both default to 0. in_f16 needs c_in % 16 == 0, c_in % 64 != 32 and an
 * INT8 (not affine) layer; out_f16 needs INT8 output (not float32) and is not available to the
 * sub-pixel entry point. Host only; HATQ_ERR_INVALID_ARG / HATQ_ERR_UNSUPPORTED.
 */
hatq_status hatq_set_operand_format(hatq_prepared *L, int in_f16, int out_f16);

/*
 * Offline preparation of a layer followed by a non-homogeneous activation
 * (Sec. general nonlinearities). The same weights, bias codes and caller-set
 * device buffers as hatq_prepare_weights, and:
 *   z = clamp(round(H~_out (M_out (.) a) / 2^n_out))      (Eq. supp_general_preactivation)
 *   u = lut[z + 127] = clamp(round(phi(s_z z) / s_u))       (Eq. supp_general_activation)
 *   x = clamp(round(H~_in,next (M_in u) / 2^n_in))         (Eq. supp_general_input_transition)
 * with s_A,c / (gamma_out s_z) ~ M_out / 2^n_out and s_u / (gamma_in,next s_y)
 * ~ M_in / 2^n_in, both pairs by the (M, n) rule of hatq_prepare_weights.
 * act: HATQ_ACT_SILU or HATQ_ACT_GELU (phi evaluated in fp64); s_z, s_u > 0;
 * the output and next-layer blocks are at most 64; INT8 output only.
 */
hatq_status hatq_prepare_weights_general(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                         float s_z, float s_u, float s_y, int act, int hb_next, hatq_prepared *out,
                                         hatq_stream stream);

/* The host half of hatq_prepare_weights_general into host arrays (sizes as for
 * hatq_prepare_weights_host; mult_in, shift_in and the 256-entry table out). */
hatq_status hatq_prepare_weights_general_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias,
                                              float s_x, float s_z, float s_u, float s_y, int act, int hb_next,
                                              int8_t *w_i8_out, uint16_t *w_f16_out, int32_t *b_int_out,
                                              int32_t *mult_out, float *s_w_out, int *shift_out,
                                              long long *mult_in_out, int *shift_in_out, int8_t *lut_out);

/*
 * Device buffer sizes of a prepared layer: w_elems = c_out * k_pad (elements
 * of w_i8 and of w_f16), ch_elems = c_out (b_int, mult, deq, s_w).
 * Returns HATQ_ERR_INVALID_ARG / HATQ_ERR_UNSUPPORTED for a bad descriptor.
 */
hatq_status hatq_prepared_sizes(const hatq_conv_desc *d, size_t *w_elems, size_t *ch_elems);

/*
 * Offline weight preparation (Eqs. double_hadamard_quantization,
 * supp_padded_wh_parameters, supp_bias_quantization, integer_fixed_point_scale;
 * Table integer_transitions).
 *   w_ohwi  host float32 [c_out][kh][kw][c_in]; bias host float32 [c_out] or NULL.
 *   s_x     scale of the INT8 operand the layer consumes (DH: in the input
 *           Hadamard basis; WH: original basis).
 *   s_y     scale of the INT8 codes the layer emits (ignored when out_f32).
 *   act     activation phi applied in the epilogue (positively homogeneous).
 *   hb_next block of the next layer's DH input transform to apply after phi
 *           (DH-to-DH / WH-to-DH transitions), 0 for none.
 *   out     caller-owned struct with its device pointers set.
 * DH: W' = W (I (x) T_in) along c_in; WH: W_bar = T_out^T W along c_out and
 * b_bar = b T_out. Per output channel s_w = max|W'|/127, w_int = round(W'/s_w),
 * b_int = round(b_bar/(s_x s_w)), rho_c = s_x s_w,c / (gamma_out gamma_in s_y),
 * M_c = round(rho_c 2^n) with the shared n chosen as the largest in [0, 62]
 * such that all M_c < 2^31 and max_c M_c A_c g_out g_next < 2^62 (A_c the
 * worst-case |accumulator|, g the unnormalized transform gains); fewer than
 * 16 multiplier bits returns HATQ_ERR_OVERFLOW. Real arithmetic is fp64 in a
 * fixed summation order. Synchronizes `stream` before returning.
 */
hatq_status hatq_prepare_weights(const hatq_conv_desc *d, const float *w_ohwi, const float *bias,
                                 float s_x, float s_y, int act, int hb_next, int out_f32,
                                 hatq_prepared *out, hatq_stream stream);

/*
 * The arithmetic of hatq_prepare_weights into caller-owned HOST buffers, with
 * no device involved (for serializing prepared layers and for checking the
 * offline step): w_i8 / w_f16 [c_out][k_pad], b_int / mult / deq / s_w
 * [c_out], *shift = n. Same arguments, rules and errors as
 * hatq_prepare_weights.
 */
hatq_status hatq_prepare_weights_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias,
                                      float s_x, float s_y, int act, int hb_next, int out_f32,
                                      int8_t *w_i8, uint16_t *w_f16, int32_t *b_int, int32_t *mult,
                                      float *deq, float *s_w, int *shift);

/*
 * Online activation transform + quantization (the activation side of
 * Eq. double_hadamard_quantization; Eq. symmetric_q; INT8 entry per
 * Eq. supp_general_input_transition).
 *   x       device NHWC, int8 codes at scale s_in (x_kind = HATQ_IN_I8) or
 *           fp16 values (HATQ_IN_F16); n*h*w*c elements, c % 16 == 0.
 *   hb      block of the unnormalized transform along c: 1 (no transform,
 *           plain requantization) or a power of two in 2..256 dividing c.
 *   s_out   > 0: static output scale; <= 0: dynamic per-tensor scale from the
 *           transformed tensor's max-abs (two passes), written to *s_used.
 *   y       device NHWC int8 codes of Q(x T) at scale s_out (or *s_used).
 *   s_used  device float, required in dynamic mode, may be NULL otherwise.
 *   workspace  device, >= 32 bytes, required in dynamic mode (reset each call).
 * FP16 entry: y = clamp(round((H~ x) / (sqrt(hb) s_out))) with an fp32
 * butterfly. INT8 entry: v = H~ x exactly in integers,
 * y = clamp(round(M_q v / 2^n_q)) with M_q / 2^n_q ~ s_in / (sqrt(hb) s_out).
 */
hatq_status hatq_quantize_act(const void *x, int x_kind, float s_in, int n, int h, int w, int c,
                              int hb, float s_out, int8_t *y, float *s_used, void *workspace,
                              hatq_stream stream);

/*
 * Convolution on INT8 operands with the fused requantize epilogue
 * (Eqs. integer_accumulation, integer_hadamard_transition):
 *   a = sum_k x_int w_int + b_int                    (exact integer)
 *   INT8 output:  y = clamp(round(H~_next phi(H~_out (M (.) a)) / 2^n))
 *   float output: y = phi(H~_out (deq (.) a))        (float32, no rounding)
 * where H~_out is applied for WH layers and H~_next when hb_next > 0; a layer
 * prepared by hatq_prepare_weights_general (SiLU / GELU) takes that entry
 * point's two-step transition instead.
 *   x   device NHWC int8 [n][h][w][c_in], the layer's operand (basis and scale s_x).
 *   y   device NHWC [n][ho][wo][c_out], int8 or float32 (L->out_f32),
 *       ho = (h + 2 pad - kh) / stride + 1 (floor), likewise wo.
 * The reduction runs on the tensor cores with the codes held exactly as fp16
 * operands and fp32 partial sums that stay below 2^24 in magnitude, moved to
 * int32 every 1024 reduction elements, so the accumulator is exact.
 * Work is enqueued only: results are complete once `stream` is synchronized
 * (check them with hatq_sync_status()).
 */
hatq_status hatq_conv2d_i8(const int8_t *x, int n, int h, int w, const hatq_prepared *L,
                           void *y, hatq_stream stream);

/*
 * One layer in one call: the activation transform/quantize of
 * hatq_quantize_act when x is not yet the layer's operand (DH: transform with
 * hb_in; WH: requantize to s_x when s_in != s_x), then hatq_conv2d_i8.
 *   x_kind   hatq_input_kind of x; s_in its scale for HATQ_IN_I8.
 *   scratch  device buffer for the INT8 operand when one is produced,
 *            >= n*h*w*c_in bytes (may be NULL when none is needed).
 */
hatq_status hatq_layer(const void *x, int x_kind, float s_in, int n, int h, int w,
                       const hatq_prepared *L, void *y, void *scratch, size_t scratch_bytes,
                       hatq_stream stream);

/*
 * hatq_layer for callers that cannot allocate device memory (code running
 * where cudaMalloc is not allowed or not available: host callbacks, plugins
 * whose host engine owns every allocation, allocator-less embeddings). The
 * paper has no counterpart: this only moves hatq_layer's scratch buffer.
 * The INT8 operand that hatq_layer would stage in `scratch` is staged in a
 * fixed device array of HATQ_NOALLOC_MAX_BYTES bytes that the library holds
 * on every device that loads it, until the process exits. An operand larger
 * than that (n*h*w*c_in bytes) returns HATQ_ERR_INVALID_ARG before any launch.
 * Nothing is allocated: no cudaMalloc/cudaFree and no allocating library call.
 * The first call on a device looks up the array's device address with that
 * device current; make that first call before any stream capture. All calls
 * share the array and it keeps the last call's contents; calls whose GPU work
 * overlaps (unordered streams) race on it. Inputs and outputs are the
 * caller's, as in hatq_layer.
 */
#define HATQ_NOALLOC_MAX_BYTES (32u << 20)
hatq_status hatq_layer_noalloc(const void *x, int x_kind, float s_in, int n, int h, int w,
                               const hatq_prepared *L, void *y, hatq_stream stream);

/* Number of kernel launches hatq_layer / hatq_conv2d_i8 make for these
 * arguments (for launch accounting), or -1 for invalid arguments. */
int hatq_layer_launches(int x_kind, float s_in, const hatq_prepared *L);

/* Message describing the calling thread's most recent failure ("" if none). */
const char *hatq_last_error(void);

/* Synchronizes `stream`, then reads and clears the device error word of the
 * current device: HATQ_ERR_TIMEOUT if a bounded wait expired, HATQ_ERR_CUDA
 * on an asynchronous CUDA error, HATQ_OK otherwise. The error word is sticky:
 * while it is set, convolution blocks that have not started return at once,
 * so work enqueued after a failure produces no output until it is read. */
hatq_status hatq_sync_status(hatq_stream stream);

/* Range-expansion profiling for the layer-wise DH/WH selection
 * (Eq. hadamard_sensitivity, Sec. profiling-based strategy selection).
 * x: device NHWC int8 codes [n][h][w][c], 16-byte aligned, c % 16 == 0;
 *    hb: the layer's input block (power of two in 2..256 dividing c).
 * maxima: device int32 [n][2], caller-owned, overwritten with max|x_k| and
 *    max|H~_hb x_k| of every image k (H~ the unnormalized block transform).
 * expands: device uint8 [n] or NULL: 1 where max|H~ x_k|^2 > hb max|x_k|^2,
 *    i.e. ||T x_k||_inf > ||x_k||_inf for the normalized transform T (exact).
 * p_l of Eq. hadamard_sensitivity is the mean of `expands` over the profiled
 * images and Eq. layerwise_hadamard_selection assigns WH iff p_l > tau_sel.
 * Stream-ordered; shape/alignment errors are returned before any launch;
 * n == 0 is a no-op. */
hatq_status hatq_profile_range(const int8_t *x, int n, int h, int w, int c, int hb, int32_t *maxima,
                               uint8_t *expands, hatq_stream stream);

/*
 * The paper's single Hadamard order per channel axis (Supp. Hadamard
 * construction; Eqs. supp_hadamard_order, supp_padded_transforms,
 * supp_padded_dh). The supported orders M_H are the Sylvester orders 2^k,
 * the Paley-I orders q + 1 (q prime, q = 3 mod 4), the Paley-II orders
 * 2 (q + 1) (q prime, q = 1 mod 4) and Kronecker products of supported
 * orders, up to 4096. Where an order has several constructions the matrix is
 * the first of Sylvester, Paley-I, Paley-II, else H~_a (x) H~_(m/a) with a the
 * smallest supported order >= 2 whose cofactor is supported.
 */
/* m(C) = the smallest supported order >= 4 ceil(C / 4) (Eq. supp_hadamard_order);
 * HATQ_ERR_UNSUPPORTED if there is none up to 4096. Host only. */
hatq_status hatq_hadamard_order(int c, int *m);
/* The unnormalized matrix H~_m (+-1 entries) into host memory, row-major
 * [m][m]; HATQ_ERR_UNSUPPORTED for an order outside M_H. Host only. */
hatq_status hatq_hadamard_matrix(int m, int8_t *h);
/*
 * A DH layer whose input side takes the paper's order m = m(c_in) over the
 * whole channel axis: W' = W (I_{KhKw} (x) P_C H_m) (Eq. supp_padded_dh, with
 * zero padding from c_in to m). d->form = HATQ_DH, d->c_in = C (the real
 * channel count), d->hb_in = 0 or m. The prepared layer consumes an operand
 * of m channels: out->d gets c_in = hb_in = m, and its device buffers are
 * sized by hatq_prepared_sizes on that descriptor. Every other argument, rule
 * and error as hatq_prepare_weights. The operand comes from the transform
 * layer of hatq_prepare_order_transform (or is already in the order-m basis).
 */
hatq_status hatq_prepare_weights_order(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                       float s_y, int act, int hb_next, int out_f32, hatq_prepared *out,
                                       hatq_stream stream);
/* The host arithmetic of hatq_prepare_weights_order into host arrays sized for
 * the order-m operand (c_out * k_pad and c_out entries). */
hatq_status hatq_prepare_weights_order_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                            float s_y, int act, int hb_next, int out_f32, int8_t *w_i8,
                                            uint16_t *w_f16, int32_t *b_int, int32_t *mult, float *deq, float *s_w,
                                            int *shift);
/*
 * The activation-side transform into the paper's order m = m(c) as a
 * bias-free 1x1 convolution (supplementary, deployment realization), run by
 * hatq_conv2d_i8 (or hatq_layer with HATQ_IN_I8) on the tensor cores: for
 * INT8 codes x at scale s_in with c channels,
 *   y_j = clamp(round(M_q (sum_{i<c} H~_m[i][j] x_i) / 2^n_q)),  j < m,
 * M_q / 2^n_q ~ s_in / (sqrt(m) s_out) by the (M, n) rule of
 * hatq_prepare_weights with the bound |sum| <= 127 c. The layer is
 * {c_in = c, c_out = m, 1x1, stride 1, form HATQ_TRANSFORM}; its device
 * buffers are sized by hatq_prepared_sizes on that descriptor (m must be a
 * multiple of 32). s_in, s_out > 0.
 */
hatq_status hatq_prepare_order_transform(int c, float s_in, float s_out, hatq_prepared *out, hatq_stream stream);

/*
 * Decoder-side operators (synthesis transforms). A transposed convolution and
 * a sub-pixel convolution are linear operators Y = X W^T like the analysis
 * convolutions (Eq. linear_operator), so the DH / WH weight transforms and
 * the integer transition apply unchanged.
 *
 * Transposed convolution with kernel kh x kw, stride s (1 or 2), padding p and
 * output padding q (0 <= q < s): input pixel (iy, ix) contributes
 * x W[:, ky, kx, :]^T to output pixel (iy s + ky - p, ix s + kx - p); the
 * output is ho = (h - 1) s - 2 p + kh + q rows (likewise wo). It runs as s^2
 * stride-1 sub-convolutions, one per output parity class (py, px): class
 * pixels (s r + py, s c + px) take the taps ky = py + p (mod s) in decreasing
 * order, kx likewise, and each class writes its pixels in place (the output
 * index remap is in the copy-out). kh, kw >= s.
 */
#define HATQ_MAX_TRANSPOSED_CLASSES 4
typedef struct {
    hatq_conv_desc d;      /* the transposed convolution (stride s, padding p, form and blocks as for a conv) */
    int out_pad;           /* q, set by the caller */
    int classes;           /* written: s * s */
    int pad_y[HATQ_MAX_TRANSPOSED_CLASSES];   /* written: the sub-convolutions' row / column offsets: class */
    int pad_x[HATQ_MAX_TRANSPOSED_CLASSES];   /* pixel r reads input row r - pad_y + j at its tap j (may be < 0) */
    hatq_prepared sub[HATQ_MAX_TRANSPOSED_CLASSES];   /* class py * s + px; the caller sets each one's six
                                                         device pointers (sizes from hatq_transposed_sizes) */
} hatq_prepared_transposed;

/* Device buffer sizes of class cls (0 <= cls < s * s) of a transposed
 * convolution: w_elems for w_i8 / w_f16, ch_elems (= c_out) for the others. */
hatq_status hatq_transposed_sizes(const hatq_conv_desc *d, int cls, size_t *w_elems, size_t *ch_elems);

/* Offline preparation of a transposed convolution: the weights are transformed
 * and quantized exactly as by hatq_prepare_weights (per-output-channel scales,
 * bias codes and (M, n) over the whole kernel), then each class's taps are
 * packed into its sub-layer. Same arguments and rules as hatq_prepare_weights;
 * out->d and out->out_pad are the caller's. Synchronizes `stream`. */
hatq_status hatq_prepare_weights_transposed(const hatq_conv_desc *d, int out_pad, const float *w_ohwi, const float *bias,
                                            float s_x, float s_y, int act, int hb_next, int out_f32,
                                            hatq_prepared_transposed *out, hatq_stream stream);

/* The transposed convolution with the fused requantize epilogue on its INT8
 * operand x [n][h][w][c_in]: y [n][ho][wo][c_out], int8 or float32 as
 * prepared. s^2 launches on `stream`. */
hatq_status hatq_conv_transpose2d_i8(const int8_t *x, int n, int h, int w, const hatq_prepared_transposed *T, void *y,
                                     hatq_stream stream);

/* hatq_conv2d_i8 followed by the sub-pixel rearrangement with factor r
 * (2 <= r <= 4): channel c r^2 + i r + j of output pixel (oy, ox) is written
 * to channel c of pixel (oy r + i, ox r + j) of y [n][ho r][wo r][c_out / r^2],
 * in the copy-out. INT8 output only; c_out and the layer's output tile must
 * hold whole 16-channel groups per sub-pixel (HATQ_ERR_UNSUPPORTED otherwise). */
hatq_status hatq_conv2d_i8_subpixel(const int8_t *x, int n, int h, int w, const hatq_prepared *L, int r, void *y,
                                    hatq_stream stream);

/*
 * Dynamic affine activation quantization (PTQ setting; Eqs. uniform_q,
 * affine_q; supplementary, affine activation quantization). Per input tensor
 * the operand v = T x (T the layer's normalized input-side block transform for
 * DH, the identity for WH) takes
 *   lo = min(min v, 0), hi = max(max v, 0), s = (hi - lo) / 255,
 *   z = clamp(round(-lo / s), 0, 255), x_int = clamp(round(v / s) + z, 0, 255)
 * (a zero range gives s = 1, z = 0), and the convolution runs on the centred
 * codes x_int - z in [-255, 255], so zero padding is a centred zero. The
 * output is dequantized: y = phi(H_out(s s_w (.) a + b_bar)).
 *
 * hatq_quantize_act_affine: x device fp16 NHWC [n][h][w][c] (c % 16 == 0), hb
 * the input-side block (1 for WH); y device int16 NHWC centred codes;
 * params device float[2] written with (s, z); workspace device >= 32 bytes
 * (reset each call). v is computed with an fp32 butterfly, so codes can differ
 * from an exact evaluation by one step where v / s lies at a rounding tie.
 */
hatq_status hatq_quantize_act_affine(const void *x, int n, int h, int w, int c, int hb, int16_t *y, float *params,
                                     void *workspace, hatq_stream stream);
/* A layer for affine activations: the weights, channel scales and transformed
 * bias of hatq_prepare_weights (any s_x: the activation scale is per input),
 * float32 output, act HATQ_ACT_NONE or HATQ_ACT_RELU, no next-layer
 * transform, c_in % 16 == 0. The bias stays real: deq holds b_bar_c / gamma_out
 * and in_affine is set. Buffers as for hatq_prepare_weights. */
hatq_status hatq_prepare_weights_affine(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, int act,
                                        hatq_prepared *out, hatq_stream stream);
/* The convolution on centred affine codes x (device int16 NHWC [n][h][w][c_in])
 * with s read from params[0] (device, as written by hatq_quantize_act_affine):
 * a = sum (x_int - z) w_int exactly (fp32 chunks of 512 products below 2^24,
 * int32 totals), y = phi(H~_out((s s_w,c / gamma_out) a + b_bar_c / gamma_out))
 * in float32, device NHWC [n][ho][wo][c_out]. */
hatq_status hatq_conv2d_affine(const int16_t *x, int n, int h, int w, const hatq_prepared *L, const float *params,
                               float *y, hatq_stream stream);

/* Layer-wise strategy selection (Eqs. hadamard_sensitivity,
 * layerwise_hadamard_selection) from the per-image indicators of
 * hatq_profile_range.
 *   expands   HOST uint8 [n], nonzero where image k's range expands; n >= 1.
 *   tau_num / tau_den   the threshold tau_sel as an exact fraction
 *             (0 <= tau_num <= tau_den, tau_den > 0; the paper uses 4 / 5).
 *   form      out: HATQ_WH when p_l > tau_sel (strict), else HATQ_DH, with
 *             p_l = (number of expanding images) / n decided exactly in
 *             integers: count * tau_den > n * tau_num.
 *   expanded  out (may be NULL): the number of expanding images, so that
 *             p_l = *expanded / n.
 * Host only, synchronous; HATQ_ERR_INVALID_ARG for a bad argument. */
hatq_status hatq_select_form(const uint8_t *expands, int n, int tau_num, int tau_den, int *form, int *expanded);

/*
 * GDN / IGDN transition (Sec. general nonlinearities, Eqs.
 * supp_general_activation, supp_general_input_scale,
 * supp_general_input_transition) for the channel-coupled activations
 * y_i = v_i / sqrt(beta_i + sum_j gamma_ij v_j^2) (IGDN: times the root),
 * v = s_z z. The layer before emits the integer preactivation z of
 * Eq. supp_general_preactivation: prepare it with hatq_prepare_weights,
 * act HATQ_ACT_NONE, hb_next 0 and output scale s_y = s_z. phi_int in
 * integers:
 *   G_ij = rint(gamma_ij s_z^2 2^e), B_i = max(1, rint(beta_i 2^e)), e the
 *     largest integer with max G <= 511 and max_i (B_i + 127^2 sum_j G_ij) < 2^31;
 *   D_i = B_i + sum_j G_ij z_j^2 (per pixel, exact);
 *   R^2 = (s_z / s_u)^2 2^e (GDN) or 2^-e (IGDN), P = rint(R^2 2^t) with the
 *     largest t in [0, 62] keeping every comparison below in 63 bits; P >= 2^15;
 *   |u_i| = the largest k <= 127 with (2k - 1)^2 D_i 2^t <= 4 P z_i^2 (GDN),
 *     (2k - 1)^2 2^t <= 4 P z_i^2 D_i (IGDN): round(R |z_i| / sqrt(D_i)) (IGDN:
 *     R |z_i| sqrt(D_i)) with ties away from zero, clamped to 127; u_i takes
 *     the sign of z_i;
 *   x = clamp(round(H~_next (M_in u) / 2^n_in), -127, 127) with
 *     s_u / (gamma_in,next s_y) ~ M_in / 2^n_in by the (M, n) rule of
 *     hatq_prepare_weights (bound 127).
 * Real arithmetic in fp64; rint rounds half to even.
 */
typedef struct {
    int c;                /* channels: 64, 128, 192 or 256 */
    int inverse;          /* 0 GDN, 1 IGDN */
    int hb_next;          /* block of the next layer's DH transform (0: none; else a power of two <= 64) */
    int e;                /* pool scale exponent */
    int t;                /* R^2 ~ P / 2^t */
    int shift_in;         /* n_in */
    long long P;
    long long mult_in;    /* M_in */
    float s_z, s_u, s_y;
    uint16_t *g_f16;      /* device [c][c] G as IEEE fp16 (exact integers <= 511); set by the caller */
    int32_t *b_pool;      /* device [c] B_i; set by the caller */
    uint64_t opaque[16];  /* the library's tensor-memory-access descriptor of g_f16 */
} hatq_prepared_gdn;

/* The arithmetic of hatq_prepare_gdn into HOST outputs: g [c][c] int32,
 * b [c] int32, and the scalars. beta [c] (> 0) and gamma [c][c] (>= 0,
 * row-major, gamma[i * c + j] = gamma_ij) are host float64. Errors:
 * HATQ_ERR_INVALID_ARG (bad argument), HATQ_ERR_UNSUPPORTED (c or hb_next
 * outside the list above), HATQ_ERR_OVERFLOW (no e, t or (M_in, n_in)
 * satisfies the bounds, or P < 2^15). */
hatq_status hatq_prepare_gdn_host(int c, const double *beta, const double *gamma, float s_z, float s_u, int inverse,
                                  float s_y, int hb_next, int32_t *g_out, int32_t *b_out, int *e_out, long long *p_out,
                                  int *t_out, long long *mult_in_out, int *shift_in_out);

/* hatq_prepare_gdn_host, then the upload of G (as fp16) and B to the caller's
 * device buffers out->g_f16 (c * c elements) and out->b_pool (c), both 16-byte
 * aligned, and the struct's other fields. Synchronizes `stream`. */
hatq_status hatq_prepare_gdn(int c, const double *beta, const double *gamma, float s_z, float s_u, int inverse,
                             float s_y, int hb_next, hatq_prepared_gdn *out, hatq_stream stream);

/* The GDN / IGDN transition on device tensors: z [n][h][w][c] INT8
 * preactivation codes in [-127, 127] (Eq. supp_general_preactivation clamps
 * to that range; -128 is outside the contract), y [n][h][w][c] the next
 * layer's INT8 operand (both 16-byte aligned, not overlapping). The pool runs on the tensor cores (the
 * squared codes in two exact fp16 limbs times G, fp32 sums below 2^24).
 * Stream-ordered; device errors surface through hatq_sync_status(). */
hatq_status hatq_gdn(const int8_t *z, int n, int h, int w, const hatq_prepared_gdn *g, int8_t *y, hatq_stream stream);

/* Failure-detection self test (the paper has no counterpart): launches one
 * thread that waits, through the same bounded mbarrier wait the convolution
 * pipeline uses, on a barrier nothing arrives at. The wait expires after
 * limit_cycles SM clock cycles (1 .. 4e9) and records the timeout in the
 * device error word, so the next hatq_sync_status() returns HATQ_ERR_TIMEOUT
 * (and clears it); convolutions enqueued before that read are skipped, as after
 * a real expiry. Stream-ordered; HATQ_ERR_INVALID_ARG for a limit out of range.
 * Nothing faults or hangs: the device stays usable. */
hatq_status hatq_selftest_wait(unsigned long long limit_cycles, hatq_stream stream);

/* Library version, (major << 16) | minor. */
int hatq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* HATQ_H */
