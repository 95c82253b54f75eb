// Host side of libhatq: the C ABI declared in include/hatq.h.
//
// Offline weight preparation follows Eqs. (double_hadamard_quantization,
// supp_padded_wh_parameters, supp_bias_quantization, integer_fixed_point_scale)
// and Table integer_transitions of the HaTQ paper; every real-valued step is
// fp64 with a fixed summation order (for output j of a block transform:
// acc = 0; acc += +-x_i for i = 0..hb-1; then acc / sqrt(hb)), so the result
// does not depend on the compiler or the machine.
#include <cuda_fp16.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "hatq.h"
#include "hatq_internal.h"

namespace {

thread_local std::string g_msg;

hatq_status fail(hatq_status st, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_msg = buf;
    return st;
}

hatq_status cuda_fail(cudaError_t e, const char *what) {
    return fail(HATQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Device error word written by kernels (bounded-wait expiry, bound checks).
__device__ int g_err_word;

int *err_word() {
    static int *ptrs[64] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    if (!ptrs[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_err_word) != cudaSuccess) return nullptr;
        ptrs[dev] = static_cast<int *>(p);
    }
    return ptrs[dev];
}

constexpr int kTileRows = 128;

bool pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }
bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
int sylvester_sign(int i, int j) { return (__builtin_popcount((unsigned)(i & j)) & 1) ? -1 : 1; }

// ------------------------------------------------------------ Hadamard orders (Supp. Hadamard construction)
//
// The supported set M_H: Sylvester orders 2^k, Paley-I orders q + 1 (q a
// prime, q = 3 mod 4), Paley-II orders 2 (q + 1) (q a prime, q = 1 mod 4) and
// Kronecker products of supported orders. Where an order has several
// constructions the matrix is the first of Sylvester, Paley-I, Paley-II, else
// H~_a (x) H~_(m/a) with a the smallest supported order >= 2 whose cofactor is
// supported (each factor by the same rule).

constexpr int kMaxOrder = 4096;

bool is_prime(int q) {
    if (q < 2) return false;
    for (int f = 2; f * f <= q; ++f)
        if (q % f == 0) return false;
    return true;
}

// 1 Sylvester, 2 Paley-I, 3 Paley-II, 0 none
int base_kind(int m) {
    if (m >= 1 && (m & (m - 1)) == 0) return 1;
    if (is_prime(m - 1) && (m - 1) % 4 == 3) return 2;
    if (m % 2 == 0 && is_prime(m / 2 - 1) && (m / 2 - 1) % 4 == 1) return 3;
    return 0;
}

const std::vector<char> &supported_table() {
    static const std::vector<char> sup = [] {
        std::vector<char> t(kMaxOrder + 1, 0);
        for (int m = 1; m <= kMaxOrder; ++m) {
            if (base_kind(m)) { t[m] = 1; continue; }
            for (int a = 2; a < m && !t[m]; ++a)
                if (m % a == 0 && t[a] && t[m / a]) t[m] = 1;
        }
        return t;
    }();
    return sup;
}

bool order_supported(int m) { return m >= 1 && m <= kMaxOrder && supported_table()[m]; }

// quadratic character modulo the prime q
std::vector<int> quadratic_character(int q) {
    std::vector<int> chi(q, -1);
    chi[0] = 0;
    for (int x = 1; x < q; ++x) chi[(long long)x * x % q] = 1;
    return chi;
}

// H~_m row-major into h (m * m entries of +-1)
void build_hadamard(int m, int8_t *h) {
    const int kind = base_kind(m);
    if (kind == 1) {
        for (int i = 0; i < m; ++i)
            for (int j = 0; j < m; ++j) h[(size_t)i * m + j] = (int8_t)sylvester_sign(i, j);
        return;
    }
    if (kind == 2) {
        // H = I + S, S = [[0, 1^T], [-1, Q]], Q[i][j] = chi(j - i)
        const int q = m - 1;
        const std::vector<int> chi = quadratic_character(q);
        for (int i = 0; i < m; ++i)
            for (int j = 0; j < m; ++j) {
                int v;
                if (i == 0) v = j == 0 ? 0 : 1;
                else if (j == 0) v = -1;
                else v = chi[((j - i) % q + q) % q];
                h[(size_t)i * m + j] = (int8_t)(v + (i == j ? 1 : 0));
            }
        return;
    }
    if (kind == 3) {
        // C = [[0, 1^T], [1, Q]] symmetric; H = C (x) [[1, 1], [1, -1]] + I (x) [[1, -1], [-1, -1]]
        const int q = m / 2 - 1, n = q + 1;
        const std::vector<int> chi = quadratic_character(q);
        const int A[2][2] = {{1, 1}, {1, -1}}, B[2][2] = {{1, -1}, {-1, -1}};
        for (int i = 0; i < n; ++i)
            for (int j = 0; j < n; ++j) {
                int c;
                if (i == 0) c = j == 0 ? 0 : 1;
                else if (j == 0) c = 1;
                else c = chi[((j - i) % q + q) % q];
                for (int k = 0; k < 2; ++k)
                    for (int l = 0; l < 2; ++l)
                        h[(size_t)(2 * i + k) * m + (2 * j + l)] = (int8_t)(c * A[k][l] + (i == j ? B[k][l] : 0));
            }
        return;
    }
    int a = 2;
    while (!(m % a == 0 && order_supported(a) && order_supported(m / a))) ++a;
    const int b = m / a;
    std::vector<int8_t> ha((size_t)a * a), hb((size_t)b * b);
    build_hadamard(a, ha.data());
    build_hadamard(b, hb.data());
    for (int i = 0; i < a; ++i)
        for (int j = 0; j < a; ++j)
            for (int k = 0; k < b; ++k)
                for (int l = 0; l < b; ++l)
                    h[(size_t)(i * b + k) * m + (j * b + l)] = (int8_t)(ha[(size_t)i * a + j] * hb[(size_t)k * b + l]);
}

// m(C) of Eq. supp_hadamard_order: the smallest supported order >= 4 ceil(C / 4); 0 if none <= kMaxOrder
int hadamard_order_of(int c) {
    if (c < 1) return 0;
    for (int m = 4 * ((c + 3) / 4); m <= kMaxOrder; ++m)
        if (order_supported(m)) return m;
    return 0;
}

// ------------------------------------------------------------ tensor maps

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// ------------------------------------------------------------ geometry

struct Geometry {
    int gather, half, cin_pad, seg, k_pad, n_t, G;
};

hatq_status check_desc(const hatq_conv_desc *d) {
    if (!d) return fail(HATQ_ERR_INVALID_ARG, "null descriptor");
    if (d->c_in < 1 || d->c_out < 32 || d->c_out % 32)
        return fail(HATQ_ERR_UNSUPPORTED, "c_in >= 1 and c_out a positive multiple of 32 are required (c_in=%d c_out=%d)",
                    d->c_in, d->c_out);
    if (d->kh < 1 || d->kw < 1 || d->kh > 16 || d->kw > 16) return fail(HATQ_ERR_INVALID_ARG, "kernel size out of range");
    if (d->stride < 1 || d->stride > 2) return fail(HATQ_ERR_UNSUPPORTED, "stride must be 1 or 2");
    if (d->pad < 0 || d->pad >= d->kh || d->pad >= d->kw) return fail(HATQ_ERR_INVALID_ARG, "padding out of range");
    if (d->form == HATQ_DH) {
        if (d->hb_out != 0) return fail(HATQ_ERR_INVALID_ARG, "a DH layer has no output block");
        const bool block = pow2(d->hb_in) && d->hb_in >= 2 && d->hb_in <= 256 && d->c_in % d->hb_in == 0;
        const bool order = d->hb_in == d->c_in && order_supported(d->hb_in);   // the paper's single order
        if (!block && !order)
            return fail(HATQ_ERR_INVALID_ARG, "DH block hb_in must be a power of two in 2..256 dividing c_in, or c_in "
                                              "itself when c_in is a supported Hadamard order");
        if (d->c_in % 16) return fail(HATQ_ERR_UNSUPPORTED, "a DH layer needs c_in % 16 == 0");
    } else if (d->form == HATQ_TRANSFORM) {
        if (d->kh != 1 || d->kw != 1 || d->stride != 1 || d->pad != 0 || d->hb_in != 0 || d->hb_out != 0)
            return fail(HATQ_ERR_INVALID_ARG, "a transform layer is a 1x1 stride-1 convolution without blocks");
        if (!order_supported(d->c_out) || d->c_out < d->c_in)
            return fail(HATQ_ERR_INVALID_ARG, "a transform layer maps c_in channels to a supported order >= c_in");
    } else if (d->form == HATQ_WH) {
        if (d->hb_in != 0) return fail(HATQ_ERR_INVALID_ARG, "a WH layer has no input block");
        if (!pow2(d->hb_out) || d->hb_out < 2 || d->hb_out > 128 || d->c_out % d->hb_out)
            return fail(HATQ_ERR_INVALID_ARG, "WH block hb_out must be a power of two in 2..128 dividing c_out");
    } else {
        return fail(HATQ_ERR_INVALID_ARG, "unknown form %d", d->form);
    }
    return HATQ_OK;
}

hatq_status geometry(const hatq_conv_desc *d, int hb_next, Geometry *g) {
    // Packed reduction order. c_in % 16 == 0: (ky, kx, ci) with ci padded to a
    // multiple of 64 per tap, except c_in % 64 == 32, where the taps follow one
    // another unpadded (a 64-wide block is two 32-channel pieces, possibly of
    // two taps) and only the total is padded to a multiple of 64. Otherwise
    // (small c_in): kernel row ky holds the kw * c_in entries (kx, ci) of one
    // contiguous input-row segment, padded with zero weights to seg (a
    // multiple of 8), rows back to back.
    g->gather = d->c_in % 16 != 0;
    g->half = !g->gather && d->c_in % 64 == 32;
    g->cin_pad = g->half ? d->c_in : (d->c_in + 63) / 64 * 64;
    g->seg = (d->kw * d->c_in + 7) / 8 * 8;
    g->k_pad = g->gather ? (d->kh * g->seg + 63) / 64 * 64 : (d->kh * d->kw * g->cin_pad + 63) / 64 * 64;
    const int hb_out = d->form == HATQ_WH ? d->hb_out : 0;
    int G = 32;
    if (hb_out > G) G = hb_out;
    if (hb_next > G) G = hb_next;
    g->G = G;
    g->n_t = 0;
    // at most 224 columns, so that two accumulator regions leave at least 64
    // TMEM columns for the fp16 A operand
    for (int nt = 224; nt >= G; nt -= 16)
        if (nt % G == 0 && d->c_out % nt == 0) { g->n_t = nt; break; }
    if (!g->n_t) return fail(HATQ_ERR_UNSUPPORTED, "no output-channel tile for c_out=%d with group %d", d->c_out, G);
    return HATQ_OK;
}

// ------------------------------------------------------------ fixed point (M, n)

// Largest n in [0, 62] with all M_c = rint(rho_c 2^n) < 2^31 and
// max_c(M_c A_c) * gain < 2^prod_bits; fewer than min_bits bits in max M is an
// error. The 64-bit epilogue takes (62, 16); the INT8-entry activation
// requantizer, a 32-bit computation, (30, 15).
hatq_status fixed_point(const std::vector<double> &rho, const std::vector<long long> &abound, long long gain,
                        std::vector<int32_t> &M, int &shift, int prod_bits = 62, int min_bits = 16) {
    for (double r : rho)
        if (!(r >= 0.0) || !std::isfinite(r)) return fail(HATQ_ERR_INVALID_ARG, "scale ratio must be finite and >= 0");
    M.assign(rho.size(), 0);
    for (int n = 62; n >= 0; --n) {
        bool ok = true;
        long long mmax = 0;
        unsigned __int128 worst = 0;
        std::vector<long long> m(rho.size());
        for (size_t c = 0; c < rho.size() && ok; ++c) {
            const double v = std::nearbyint(std::ldexp(rho[c], n));
            if (v >= 2147483648.0) { ok = false; break; }
            m[c] = (long long)v;
            if (m[c] > mmax) mmax = m[c];
            const unsigned __int128 w = (unsigned __int128)m[c] * (unsigned __int128)abound[c];
            if (w > worst) worst = w;
        }
        if (!ok) continue;
        if (worst * (unsigned __int128)gain >= ((unsigned __int128)1 << prod_bits)) continue;
        if (mmax < (1LL << (min_bits - 1)))
            return fail(HATQ_ERR_OVERFLOW, "fewer than %d bits of multiplier precision", min_bits);
        for (size_t c = 0; c < rho.size(); ++c) M[c] = (int32_t)m[c];
        shift = n;
        return HATQ_OK;
    }
    return fail(HATQ_ERR_OVERFLOW, "no shift satisfies the multiplier and overflow bounds");
}

// Normalized transform of one contiguous hb-block x into y (element j at
// y[j * ystep]) in the fixed order: acc = 0; acc += +-x_i, i = 0..hb-1; acc / sqrt(hb).
void block_transform(const double *x, double *y, int hb, long long ystep) {
    const double sq = std::sqrt((double)hb);
    for (int j = 0; j < hb; ++j) {
        double acc = 0.0;
        for (int i = 0; i < hb; ++i) acc += sylvester_sign(i, j) > 0 ? x[i] : -x[i];
        y[j * ystep] = acc / sq;
    }
}

uint16_t f16_bits(int v) {
    const __half h = __float2half_rn((float)v);
    uint16_t b;
    std::memcpy(&b, &h, 2);
    return b;
}

void choose_mtile(int ho, int wo, int stride, int *tw, int *th) {
    long long best = -1;
    for (int t = 128; t >= 8; t >>= 1) {
        const int h = 128 / t;
        if (t * stride > 256 || h * stride > 256) continue;
        const long long area = (long long)((wo + t - 1) / t) * t * (long long)((ho + h - 1) / h) * h;
        if (best < 0 || area < best) { best = area; *tw = t; *th = h; }
    }
}

// Bytes of one row of a small-channel layer's TMA window box: the window's
// win_w * c bytes starting anywhere inside a 16-byte granule, rounded up to 16.
int window_box_bytes(int tw, int stride, int kw, int c) { return (((tw - 1) * stride + kw) * c + 15 + 15) & ~15; }

// Tile shape of a small-channel layer whose input window is loaded as one TMA
// box per tile (box row <= 256 bytes and rows <= 256), or false when none fits
// (the window is then staged by the converter warps).
bool choose_window_tile(int ho, int wo, int stride, int kh, int kw, int c, int *tw, int *th) {
    long long best = -1;
    for (int t = 128; t >= 8; t >>= 1) {
        const int h = 128 / t;
        if (window_box_bytes(t, stride, kw, c) > 256 || (h - 1) * stride + kh > 256) continue;
        const long long area = (long long)((wo + t - 1) / t) * t * (long long)((ho + h - 1) / h) * h;
        if (best < 0 || area < best) { best = area; *tw = t; *th = h; }
    }
    return best >= 0;
}

hatq_status validate_prepare(const hatq_conv_desc *d, const float *w_ohwi, float s_x, float s_y, int act,
                                    int hb_next, int out_f32, Geometry *g) {
    hatq_status st = check_desc(d);
    if (st != HATQ_OK) return st;
    if (d->form == HATQ_TRANSFORM)
        return fail(HATQ_ERR_INVALID_ARG, "transform layers are prepared with hatq_prepare_order_transform");
    if (!w_ohwi) return fail(HATQ_ERR_INVALID_ARG, "null weights");
    if (!(s_x > 0.f) || !std::isfinite(s_x)) return fail(HATQ_ERR_INVALID_ARG, "s_x must be positive");
    if (!out_f32 && (!(s_y > 0.f) || !std::isfinite(s_y))) return fail(HATQ_ERR_INVALID_ARG, "s_y must be positive");
    if (act != HATQ_ACT_NONE && act != HATQ_ACT_RELU && act != HATQ_ACT_SILU && act != HATQ_ACT_GELU)
        return fail(HATQ_ERR_INVALID_ARG, "unknown activation");
    if (hb_next != 0 && (!pow2(hb_next) || hb_next < 2 || hb_next > 128 || d->c_out % hb_next))
        return fail(HATQ_ERR_INVALID_ARG, "hb_next must be 0 or a power of two in 2..128 dividing c_out");
    if (out_f32 && hb_next) return fail(HATQ_ERR_INVALID_ARG, "a float32 output has no next-layer transform");
    return geometry(d, hb_next, g);
}

bool general_act(int act) { return act == HATQ_ACT_SILU || act == HATQ_ACT_GELU; }

// phi of Sec. general nonlinearities in fp64: SiLU v / (1 + e^-v), GELU v (1 + erf(v / sqrt 2)) / 2.
double phi(int act, double v) {
    if (act == HATQ_ACT_SILU) return v / (1.0 + std::exp(-v));
    return 0.5 * v * (1.0 + std::erf(v / std::sqrt(2.0)));
}

// The second half of a general transition: preactivation / activation scales
// in, table and input-side fixed point out (Eqs. supp_general_activation,
// supp_general_input_scale).
struct GeneralParams {
    float s_z = 0.f, s_u = 0.f;
    long long mult_in = 0;
    int shift_in = 0;
    int8_t lut[256] = {};
};

hatq_status validate_general(const hatq_conv_desc *d, int act, int hb_next, int out_f32, float s_z, float s_u) {
    if (!general_act(act)) return fail(HATQ_ERR_INVALID_ARG, "the general transition takes HATQ_ACT_SILU or HATQ_ACT_GELU");
    if (out_f32) return fail(HATQ_ERR_INVALID_ARG, "the general transition emits INT8 codes");
    if (!(s_z > 0.f) || !std::isfinite(s_z) || !(s_u > 0.f) || !std::isfinite(s_u))
        return fail(HATQ_ERR_INVALID_ARG, "s_z and s_u must be positive");
    const int hb_out = d->form == HATQ_WH ? d->hb_out : 0;
    if (hb_out > 64 || hb_next > 64)
        return fail(HATQ_ERR_UNSUPPORTED, "the general transition supports output and next-layer blocks up to 64");
    return HATQ_OK;
}

// The descriptor of the operand a layer consumes: for a DH layer in the
// paper's single order (order > 0) the operand has m = order channels and the
// block is the whole axis; otherwise the caller's descriptor.
hatq_status operand_desc(const hatq_conv_desc *d, int order, hatq_conv_desc *op) {
    if (!d) return fail(HATQ_ERR_INVALID_ARG, "null descriptor");
    *op = *d;
    if (!order) {
        if (d->form == HATQ_DH && !pow2(d->hb_in))
            return fail(HATQ_ERR_INVALID_ARG, "a paper-order DH layer is prepared with hatq_prepare_weights_order");
        return HATQ_OK;
    }
    if (d->form != HATQ_DH) return fail(HATQ_ERR_UNSUPPORTED, "the paper's single order is implemented for DH layers");
    if (d->c_in < 1 || (d->hb_in != 0 && d->hb_in != order))
        return fail(HATQ_ERR_INVALID_ARG, "hb_in of a paper-order layer must be 0 or m(c_in) = %d", order);
    op->c_in = order;
    op->hb_in = order;
    return HATQ_OK;
}

hatq_status prepare_core(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x, float s_y,
                         int act, int hb_next, int out_f32, GeneralParams *gen, int order, int8_t *w_i8_out,
                         uint16_t *w_f16_out, int32_t *b_int_out, int32_t *mult_out, float *deq_out, float *s_w_out,
                         int *shift_out, double *bbar_out = nullptr) {
    hatq_conv_desc dop;
    hatq_status st = operand_desc(d, order, &dop);
    if (st != HATQ_OK) return st;
    const int c_src = d->c_in;                      // channels of the real-valued weights
    d = &dop;
    Geometry g;
    st = validate_prepare(d, w_ohwi, s_x, s_y, act, hb_next, out_f32, &g);
    if (st != HATQ_OK) return st;
    if (general_act(act) != (gen != nullptr))
        return fail(HATQ_ERR_INVALID_ARG, "SiLU / GELU layers are prepared with hatq_prepare_weights_general");
    if (gen && (st = validate_general(d, act, hb_next, out_f32, gen->s_z, gen->s_u)) != HATQ_OK) return st;
    if (!w_i8_out || !w_f16_out || !b_int_out || !mult_out || !deq_out || !s_w_out || !shift_out)
        return fail(HATQ_ERR_INVALID_ARG, "null output buffer");
    const int co = d->c_out, ci = d->c_in, taps = d->kh * d->kw;
    const long long per_o = (long long)taps * ci;
    // 1. Hadamard-domain weights and bias (fp64)
    std::vector<double> wp((size_t)co * per_o);
    std::vector<double> bbar(co, 0.0);
    if (bias)
        for (int o = 0; o < co; ++o) bbar[o] = (double)bias[o];
    if (order) {
        // Eq. supp_padded_dh: W' = W (I (x) P_C H_m), output j of a tap in the fixed order
        // acc = 0; acc += +-w_i, i = 0..C-1; acc / sqrt(m)
        std::vector<int8_t> h((size_t)order * order);
        build_hadamard(order, h.data());
        const double sq = std::sqrt((double)order);
        for (long long r = 0; r < (long long)co * taps; ++r)
            for (int j = 0; j < order; ++j) {
                double acc = 0.0;
                for (int i = 0; i < c_src; ++i) {
                    const double x = (double)w_ohwi[r * c_src + i];
                    acc += h[(size_t)i * order + j] > 0 ? x : -x;
                }
                wp[r * ci + j] = acc / sq;
            }
    } else if (d->form == HATQ_DH) {
        const int hb = d->hb_in;
        for (long long r = 0; r < (long long)co * taps; ++r)
            for (int blk = 0; blk < ci / hb; ++blk) {
                double x[256];
                for (int i = 0; i < hb; ++i) x[i] = (double)w_ohwi[r * ci + blk * hb + i];
                block_transform(x, &wp[r * ci + blk * hb], hb, 1);
            }
    } else {
        const int hb = d->hb_out;
        for (long long t = 0; t < per_o; ++t)            // (tap, ci) column, transform along c_out
            for (int blk = 0; blk < co / hb; ++blk) {
                double x[128];
                for (int i = 0; i < hb; ++i) x[i] = (double)w_ohwi[(long long)(blk * hb + i) * per_o + t];
                block_transform(x, &wp[(long long)(blk * hb) * per_o + t], hb, per_o);
            }
        std::vector<double> b0 = bbar;
        for (int blk = 0; blk < co / hb; ++blk) block_transform(&b0[blk * hb], &bbar[blk * hb], hb, 1);
    }
    if (bbar_out)
        for (int o = 0; o < co; ++o) bbar_out[o] = bbar[o];
    // 2. channel-wise symmetric weight quantization, bias codes, bounds
    std::vector<double> s_a(co), rho(co);
    std::vector<long long> abound(co);
    std::memset(w_i8_out, 0, (size_t)co * g.k_pad);
    for (size_t k = 0; k < (size_t)co * g.k_pad; ++k) w_f16_out[k] = f16_bits(0);
    const double sx = (double)s_x, sy = (double)s_y;
    for (int o = 0; o < co; ++o) {
        const double *row = &wp[(size_t)o * per_o];
        double m = 0.0;
        for (long long k = 0; k < per_o; ++k) m = std::fmax(m, std::fabs(row[k]));
        const double sw = m > 0.0 ? m / 127.0 : 1.0;
        long long sum_abs = 0;
        for (int tap = 0; tap < taps; ++tap)
            for (int c = 0; c < ci; ++c) {
                double q = std::nearbyint(row[(long long)tap * ci + c] / sw);
                q = q < -127.0 ? -127.0 : (q > 127.0 ? 127.0 : q);
                const int qi = (int)q;
                sum_abs += qi < 0 ? -qi : qi;
                const long long k = g.gather ? (long long)(tap / d->kw) * g.seg + (tap % d->kw) * ci + c
                                             : (long long)tap * g.cin_pad + c;
                w_i8_out[(size_t)o * g.k_pad + k] = (int8_t)qi;
                w_f16_out[(size_t)o * g.k_pad + k] = f16_bits(qi);
            }
        s_a[o] = sx * sw;
        const double bq = std::nearbyint(bbar[o] / s_a[o]);
        if (!(std::fabs(bq) < 1073741824.0)) return fail(HATQ_ERR_OVERFLOW, "bias code of channel %d out of range", o);
        b_int_out[o] = (int32_t)bq;
        abound[o] = 127LL * sum_abs + (long long)std::llabs((long long)b_int_out[o]);
        if (abound[o] >= (1LL << 31)) return fail(HATQ_ERR_OVERFLOW, "int32 accumulator bound exceeded in channel %d", o);
        s_w_out[o] = (float)sw;
    }
    // 3. requantization (Eq. integer_fixed_point_scale; gammas of Table integer_transitions)
    const double g_out = d->form == HATQ_WH ? std::sqrt((double)d->hb_out) : 1.0;
    const double g_in = hb_next ? std::sqrt((double)hb_next) : 1.0;
    for (int o = 0; o < co; ++o) deq_out[o] = (float)(s_a[o] / g_out);
    *shift_out = 0;
    if (out_f32) {
        for (int o = 0; o < co; ++o) mult_out[o] = 0;
        return HATQ_OK;
    }
    std::vector<int32_t> mult;
    int shift = 0;
    if (gen) {
        // Eq. supp_general_output_scale: s_A,c / (gamma_out s_z), M_out applied before H_out
        const double sz = (double)gen->s_z, su = (double)gen->s_u;
        for (int o = 0; o < co; ++o) rho[o] = s_a[o] / (g_out * sz);
        if ((st = fixed_point(rho, abound, d->form == HATQ_WH ? d->hb_out : 1, mult, shift)) != HATQ_OK) return st;
        // Eq. supp_general_activation as a table over z = -127..127
        for (int z = -127; z <= 127; ++z) {
            double u = std::nearbyint(phi(act, sz * (double)z) / su);
            u = u < -127.0 ? -127.0 : (u > 127.0 ? 127.0 : u);
            gen->lut[z + 127] = (int8_t)u;
        }
        gen->lut[255] = 0;
        // Eq. supp_general_input_scale: s_u / (gamma_in,next s_x,next)
        std::vector<int32_t> m_in;
        int n_in = 0;
        if ((st = fixed_point({su / (g_in * sy)}, {127LL}, hb_next ? hb_next : 1, m_in, n_in)) != HATQ_OK) return st;
        gen->mult_in = m_in[0];
        gen->shift_in = n_in;
    } else {
        const double alpha = g_out * g_in;
        for (int o = 0; o < co; ++o) rho[o] = s_a[o] / (alpha * sy);
        const long long gain = (long long)(d->form == HATQ_WH ? d->hb_out : 1) * (hb_next ? hb_next : 1);
        if ((st = fixed_point(rho, abound, gain, mult, shift)) != HATQ_OK) return st;
    }
    for (int o = 0; o < co; ++o) mult_out[o] = mult[o];
    *shift_out = shift;
    return HATQ_OK;
}

}  // namespace

hatq_status hatq::report(hatq_status st, const char *msg) { return fail(st, "%s", msg); }

extern "C" {

int hatq_version(void) { return (0 << 16) | 1; }

const char *hatq_last_error(void) { return g_msg.c_str(); }

hatq_status hatq_prepared_sizes(const hatq_conv_desc *d, size_t *w_elems, size_t *ch_elems) {
    hatq_status st = check_desc(d);
    if (st != HATQ_OK) return st;
    Geometry g;
    if ((st = geometry(d, 0, &g)) != HATQ_OK) return st;
    if (w_elems) *w_elems = (size_t)d->c_out * g.k_pad;
    if (ch_elems) *ch_elems = (size_t)d->c_out;
    return HATQ_OK;
}

hatq_status hatq_prepare_weights_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                      float s_y, int act, int hb_next, int out_f32, int8_t *w_i8_out,
                                      uint16_t *w_f16_out, int32_t *b_int_out, int32_t *mult_out, float *deq_out,
                                      float *s_w_out, int *shift_out) {
    return prepare_core(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, nullptr, 0, w_i8_out, w_f16_out, b_int_out,
                        mult_out, deq_out, s_w_out, shift_out);
}

hatq_status hatq_prepare_weights_order_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                            float s_y, int act, int hb_next, int out_f32, int8_t *w_i8_out,
                                            uint16_t *w_f16_out, int32_t *b_int_out, int32_t *mult_out,
                                            float *deq_out, float *s_w_out, int *shift_out) {
    const int m = d ? hadamard_order_of(d->c_in) : 0;
    if (d && !m) return fail(HATQ_ERR_UNSUPPORTED, "no supported Hadamard order for c_in=%d", d->c_in);
    return prepare_core(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, nullptr, m, w_i8_out, w_f16_out, b_int_out,
                        mult_out, deq_out, s_w_out, shift_out);
}

hatq_status hatq_prepare_weights_general_host(const hatq_conv_desc *d, const float *w_ohwi, const float *bias,
                                              float s_x, float s_z, float s_u, float s_y, int act, int hb_next,
                                              int8_t *w_i8_out, uint16_t *w_f16_out, int32_t *b_int_out,
                                              int32_t *mult_out, float *s_w_out, int *shift_out,
                                              long long *mult_in_out, int *shift_in_out, int8_t *lut_out) {
    if (!mult_in_out || !shift_in_out || !lut_out) return fail(HATQ_ERR_INVALID_ARG, "null output buffer");
    const int co = d ? d->c_out : 0;
    std::vector<float> deq(co > 0 ? co : 1);
    GeneralParams gen;
    gen.s_z = s_z;
    gen.s_u = s_u;
    hatq_status st = prepare_core(d, w_ohwi, bias, s_x, s_y, act, hb_next, 0, &gen, 0, w_i8_out, w_f16_out, b_int_out,
                                  mult_out, deq.data(), s_w_out, shift_out);
    if (st != HATQ_OK) return st;
    *mult_in_out = gen.mult_in;
    *shift_in_out = gen.shift_in;
    std::memcpy(lut_out, gen.lut, 256);
    return HATQ_OK;
}

}  // extern "C"

namespace {

// Host arrays of a prepared layer in the library's packed layout.
struct HostLayer {
    std::vector<int8_t> w_i8;
    std::vector<uint16_t> w_f16;
    std::vector<int32_t> b_int, mult;
    std::vector<float> deq, s_w;
    int shift = 0;
    HostLayer(int co, int k_pad) : w_i8((size_t)co * k_pad), w_f16((size_t)co * k_pad), b_int(co), mult(co), deq(co),
                                   s_w(co) {}
};

hatq_status check_out_buffers(const hatq_prepared *out) {
    if (!out) return fail(HATQ_ERR_INVALID_ARG, "null output struct");
    if (!out->w_i8 || !out->w_f16 || !out->b_int || !out->mult || !out->deq || !out->s_w)
        return fail(HATQ_ERR_INVALID_ARG, "prepared-layer device buffers must be set before preparation");
    if (!aligned16(out->w_i8) || !aligned16(out->w_f16) || !aligned16(out->b_int) || !aligned16(out->mult) ||
        !aligned16(out->deq) || !aligned16(out->s_w))
        return fail(HATQ_ERR_INVALID_ARG, "prepared-layer device buffers must be 16-byte aligned");
    return HATQ_OK;
}

// Copies the host arrays to the caller's device buffers, encodes the weight
// tensor map and fills the struct (dop: the descriptor of the operand).
hatq_status upload_layer(const hatq_conv_desc &dop, const Geometry &g, const HostLayer &hl, int act, int hb_next,
                         int out_f32, float s_x, float s_y, const GeneralParams *gen, hatq_prepared *out,
                         hatq_stream stream) {
    const int co = dop.c_out;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e;
    if ((e = cudaMemcpyAsync(out->w_i8, hl.w_i8.data(), hl.w_i8.size(), cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->w_f16, hl.w_f16.data(), hl.w_f16.size() * 2, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->b_int, hl.b_int.data(), co * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->mult, hl.mult.data(), co * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->deq, hl.deq.data(), co * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->s_w, hl.s_w.data(), co * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(e, "upload of prepared weights");
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return cuda_fail(e, "upload of prepared weights");
    // weight tensor map: [c_out][k_pad] fp16, 64 x n_t box, 128-byte swizzle
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(HATQ_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    CUtensorMap tm;
    const cuuint64_t dims[2] = {(cuuint64_t)g.k_pad, (cuuint64_t)co};
    const cuuint64_t strides[1] = {(cuuint64_t)g.k_pad * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)g.n_t};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, out->w_f16, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HATQ_ERR_CUDA, "weight tensor map encoding failed (%d)", (int)r);
    static_assert(sizeof(CUtensorMap) <= sizeof(out->opaque), "opaque area too small");
    std::memcpy(out->opaque, &tm, sizeof tm);

    out->d = dop;
    out->act = act;
    out->hb_next = hb_next;
    out->out_f32 = out_f32 ? 1 : 0;
    out->shift = hl.shift;
    out->k_pad = g.k_pad;
    out->gather = g.gather;
    out->s_x = s_x;
    out->s_y = out_f32 ? 0.f : s_y;
    out->s_z = gen ? gen->s_z : 0.f;
    out->s_u = gen ? gen->s_u : 0.f;
    out->shift_in = gen ? gen->shift_in : 0;
    out->in_affine = 0;
    out->in_f16 = 0;
    out->out_f16 = 0;
    out->mult_in = gen ? gen->mult_in : 0;
    if (gen) std::memcpy(out->lut, gen->lut, sizeof out->lut);
    else std::memset(out->lut, 0, sizeof out->lut);
    return HATQ_OK;
}

hatq_status prepare_device(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x, float s_y,
                           int act, int hb_next, int out_f32, GeneralParams *gen, int order, hatq_prepared *out,
                           hatq_stream stream) {
    hatq_conv_desc dop;
    hatq_status st = operand_desc(d, order, &dop);
    if (st != HATQ_OK) return st;
    Geometry g;
    if ((st = validate_prepare(&dop, w_ohwi, s_x, s_y, act, hb_next, out_f32, &g)) != HATQ_OK) return st;
    if ((st = check_out_buffers(out)) != HATQ_OK) return st;
    HostLayer hl(dop.c_out, g.k_pad);
    st = prepare_core(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, gen, order, hl.w_i8.data(), hl.w_f16.data(),
                      hl.b_int.data(), hl.mult.data(), hl.deq.data(), hl.s_w.data(), &hl.shift);
    if (st != HATQ_OK) return st;
    return upload_layer(dop, g, hl, act, hb_next, out_f32, s_x, s_y, gen, out, stream);
}

// The activation-side transform of the paper's order m = m(c) as a 1x1
// convolution (Sec. deployment realization): c input channels (codes in the
// original basis at s_in), m output channels, weights w[j][i] = H~_m[i][j],
// zero bias, one multiplier M_q / 2^n_q ~ s_in / (sqrt(m) s_out) by the
// (M, n) rule over |y| <= 127 c.
hatq_status transform_core(int c, float s_in, float s_out, hatq_conv_desc *dt, Geometry *g, HostLayer **out) {
    const int m = hadamard_order_of(c);
    if (!m) return fail(HATQ_ERR_UNSUPPORTED, "no supported Hadamard order for c=%d", c);
    if (!(s_in > 0.f) || !std::isfinite(s_in) || !(s_out > 0.f) || !std::isfinite(s_out))
        return fail(HATQ_ERR_INVALID_ARG, "s_in and s_out must be positive");
    *dt = hatq_conv_desc{c, m, 1, 1, 1, 0, HATQ_TRANSFORM, 0, 0};
    hatq_status st = check_desc(dt);
    if (st != HATQ_OK) return st;
    if ((st = geometry(dt, 0, g)) != HATQ_OK) return st;
    std::vector<int8_t> h((size_t)m * m);
    build_hadamard(m, h.data());
    HostLayer *hl = new HostLayer(m, g->k_pad);
    for (int j = 0; j < m; ++j) {
        for (int k = 0; k < g->k_pad; ++k) hl->w_f16[(size_t)j * g->k_pad + k] = f16_bits(0);
        for (int i = 0; i < c; ++i) {       // 1x1: reduction index i in both packings
            hl->w_i8[(size_t)j * g->k_pad + i] = h[(size_t)i * m + j];
            hl->w_f16[(size_t)j * g->k_pad + i] = f16_bits(h[(size_t)i * m + j]);
        }
    }
    std::vector<int32_t> M;
    const double rho = (double)s_in / (std::sqrt((double)m) * (double)s_out);
    if ((st = fixed_point(std::vector<double>(1, rho), std::vector<long long>(1, 127LL * c), 1, M, hl->shift)) !=
        HATQ_OK) {
        delete hl;
        return st;
    }
    for (int j = 0; j < m; ++j) {
        hl->mult[j] = M[0];
        hl->b_int[j] = 0;
        hl->deq[j] = 0.f;
        hl->s_w[j] = 1.f;
    }
    *out = hl;
    return HATQ_OK;
}

}  // namespace

extern "C" {

hatq_status hatq_prepare_weights(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                 float s_y, int act, int hb_next, int out_f32, hatq_prepared *out,
                                 hatq_stream stream) {
    return prepare_device(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, nullptr, 0, out, stream);
}

hatq_status hatq_hadamard_order(int c, int *m) {
    if (!m) return fail(HATQ_ERR_INVALID_ARG, "null output");
    if (c < 1) return fail(HATQ_ERR_INVALID_ARG, "c must be positive");
    *m = hadamard_order_of(c);
    if (!*m) return fail(HATQ_ERR_UNSUPPORTED, "no supported Hadamard order >= 4 ceil(c / 4) up to %d", kMaxOrder);
    return HATQ_OK;
}

hatq_status hatq_hadamard_matrix(int m, int8_t *h) {
    if (!h) return fail(HATQ_ERR_INVALID_ARG, "null output");
    if (!order_supported(m)) return fail(HATQ_ERR_UNSUPPORTED, "order %d is not supported", m);
    build_hadamard(m, h);
    return HATQ_OK;
}

hatq_status hatq_prepare_weights_order(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                       float s_y, int act, int hb_next, int out_f32, hatq_prepared *out,
                                       hatq_stream stream) {
    const int m = d ? hadamard_order_of(d->c_in) : 0;
    if (d && !m) return fail(HATQ_ERR_UNSUPPORTED, "no supported Hadamard order for c_in=%d", d->c_in);
    return prepare_device(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, nullptr, m, out, stream);
}

hatq_status hatq_prepare_order_transform(int c, float s_in, float s_out, hatq_prepared *out, hatq_stream stream) {
    hatq_status st = check_out_buffers(out);
    if (st != HATQ_OK) return st;
    hatq_conv_desc dt;
    Geometry g;
    HostLayer *hl = nullptr;
    if ((st = transform_core(c, s_in, s_out, &dt, &g, &hl)) != HATQ_OK) return st;
    st = upload_layer(dt, g, *hl, HATQ_ACT_NONE, 0, 0, s_in, s_out, nullptr, out, stream);
    delete hl;
    return st;
}

hatq_status hatq_prepare_weights_general(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, float s_x,
                                         float s_z, float s_u, float s_y, int act, int hb_next, hatq_prepared *out,
                                         hatq_stream stream) {
    GeneralParams gen;
    gen.s_z = s_z;
    gen.s_u = s_u;
    return prepare_device(d, w_ohwi, bias, s_x, s_y, act, hb_next, 0, &gen, 0, out, stream);
}

hatq_status hatq_quantize_act(const void *x, int x_kind, float s_in, int n, int h, int w, int c, int hb, float s_out,
                              int8_t *y, float *s_used, void *workspace, hatq_stream stream) {
    if (n == 0 && h >= 0 && w >= 0 && c >= 0) return HATQ_OK;        // empty batch: nothing to do
    if (!x || !y) return fail(HATQ_ERR_INVALID_ARG, "null input or output");
    if (!aligned16(x) || !aligned16(y)) return fail(HATQ_ERR_INVALID_ARG, "input and output must be 16-byte aligned");
    if (x_kind != HATQ_IN_I8 && x_kind != HATQ_IN_F16) return fail(HATQ_ERR_INVALID_ARG, "x_kind must be I8 or F16");
    if (n < 0 || h < 0 || w < 0 || c < 16 || c % 16) return fail(HATQ_ERR_INVALID_ARG, "shape must be n,h,w >= 0, c % 16 == 0");
    if (!pow2(hb) || hb > 256 || c % hb) return fail(HATQ_ERR_INVALID_ARG, "hb must be a power of two <= 256 dividing c");
    const bool dynamic = !(s_out > 0.f);
    if (x_kind == HATQ_IN_I8 && !(s_in > 0.f)) return fail(HATQ_ERR_INVALID_ARG, "s_in must be positive");
    if (dynamic && (!s_used || !workspace)) return fail(HATQ_ERR_INVALID_ARG, "dynamic mode needs s_used and workspace");
    if (dynamic && !aligned16(workspace)) return fail(HATQ_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
    const long long total = (long long)n * h * w * c;
    hatq::ActQuantArgs a{};
    a.x = x;
    a.y = y;
    a.total = total;
    a.hb = hb;
    a.f16 = x_kind == HATQ_IN_F16;
    a.err = err_word();
    if (!a.err) return fail(HATQ_ERR_CUDA, "no CUDA device");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (total == 0) return HATQ_OK;
    cudaError_t e;
    if (dynamic) {
        a.dyn = static_cast<hatq::DynParams *>(workspace);
        e = hatq::launch_act_dynamic(a, s_in, s_used, s);
    } else {
        if (a.f16) {
            a.inv = (float)(1.0 / (std::sqrt((double)hb) * (double)s_out));
        } else {
            const double rho = (double)s_in / (std::sqrt((double)hb) * (double)s_out);
            std::vector<int32_t> M;
            int shift = 0;
            hatq_status st = fixed_point({rho}, {127LL * hb}, 1, M, shift, 30, 15);
            if (st != HATQ_OK) return st;
            a.mult = M[0];
            a.shift = shift;
        }
        e = hatq::launch_act_quant(a, s);
    }
    if (e != cudaSuccess) return cuda_fail(e, "activation quantization launch");
    return HATQ_OK;
}

}  // extern "C"

namespace {

// Where a launch's output pixels come from and go to (see ConvArgs): a plain
// convolution, one output parity class of a transposed convolution, or a
// convolution followed by the sub-pixel rearrangement.
struct OutGrid {
    int pad_y, pad_x, ho, wo, y_h, y_w, ostride, ooy, oox, d2s;
};

hatq_status conv_launch(const void *x, int n, int h, int w, const hatq_prepared *L, void *y, hatq_stream stream,
                        const OutGrid *og, const float *affine_s = nullptr) {
    if (!L) return fail(HATQ_ERR_INVALID_ARG, "null layer");
    if (n == 0 && h >= 1 && w >= 1) return HATQ_OK;                    // empty batch: nothing to do
    if (!x || !y) return fail(HATQ_ERR_INVALID_ARG, "null argument");
    if (!aligned16(x) || !aligned16(y)) return fail(HATQ_ERR_INVALID_ARG, "input and output must be 16-byte aligned");
    const hatq_conv_desc *d = &L->d;
    hatq_status st = check_desc(d);
    if (st != HATQ_OK) return st;
    if (n < 0 || h < 1 || w < 1) return fail(HATQ_ERR_INVALID_ARG, "bad input shape");
    int ho, wo;
    if (og) {
        ho = og->ho;
        wo = og->wo;
    } else {
        ho = (h + 2 * d->pad - d->kh) / d->stride + 1;
        wo = (w + 2 * d->pad - d->kw) / d->stride + 1;
        if (h + 2 * d->pad < d->kh || w + 2 * d->pad < d->kw || ho < 1 || wo < 1)
            return fail(HATQ_ERR_INVALID_ARG, "input smaller than the kernel");
    }
    if (ho < 1 || wo < 1) return HATQ_OK;
    if ((long long)n * h * w * d->c_in >= (1LL << 40)) return fail(HATQ_ERR_UNSUPPORTED, "input too large");
    if ((L->in_affine != 0) != (affine_s != nullptr))
        return fail(HATQ_ERR_INVALID_ARG, L->in_affine ? "a layer prepared for affine activations runs through "
                                                         "hatq_conv2d_affine"
                                                       : "hatq_conv2d_affine needs a layer from "
                                                         "hatq_prepare_weights_affine");
    if (n == 0) return HATQ_OK;
    Geometry g;
    if ((st = geometry(d, L->hb_next, &g)) != HATQ_OK) return st;
    if (g.k_pad != L->k_pad || g.gather != L->gather) return fail(HATQ_ERR_INVALID_ARG, "prepared layer is inconsistent");
    if ((long long)n * ((ho + 0) * (long long)wo) > (1LL << 31)) return fail(HATQ_ERR_UNSUPPORTED, "too many output pixels");

    hatq::ConvArgs a{};
    a.n = n; a.h = h; a.w = w; a.c = d->c_in;
    a.ho = ho; a.wo = wo; a.co = d->c_out;
    a.kh = d->kh; a.kw = d->kw; a.stride = d->stride;
    a.pad_y = og ? og->pad_y : d->pad;
    a.pad_x = og ? og->pad_x : d->pad;
    a.y_h = og ? og->y_h : ho;
    a.y_w = og ? og->y_w : wo;
    a.ostride = og ? og->ostride : 1;
    a.ooy = og ? og->ooy : 0;
    a.oox = og ? og->oox : 0;
    a.d2s = og ? og->d2s : 0;
    // the small-channel loader takes its window by TMA when the input rows are 16-byte multiples
    // (the tensor map's stride rule) and a tile shape's window fits one box
    a.win_tma = g.gather && ((long long)w * d->c_in) % 16 == 0 &&
                choose_window_tile(ho, wo, d->stride, d->kh, d->kw, d->c_in, &a.tw, &a.th);
    if (!a.win_tma) choose_mtile(ho, wo, d->stride, &a.tw, &a.th);
    a.tw_log2 = __builtin_ctz((unsigned)a.tw);
    a.tiles_w = (wo + a.tw - 1) / a.tw;
    a.tiles_h = (ho + a.th - 1) / a.th;
    if ((long long)n * a.tiles_w * a.tiles_h >= (1LL << 31)) return fail(HATQ_ERR_UNSUPPORTED, "grid too large");
    a.n_t = g.n_t;
    if (a.d2s) {
        const int r2 = a.d2s * a.d2s;
        if (L->out_f32) return fail(HATQ_ERR_UNSUPPORTED, "the sub-pixel rearrangement is built for INT8 output");
        if (L->hb_next)   // the next layer's channel axis is the rearranged one, not this layer's output axis
            return fail(HATQ_ERR_UNSUPPORTED, "a sub-pixel layer takes no fused next-layer transform");
        if (d->c_out % r2 || a.n_t % (16 * r2))
            return fail(HATQ_ERR_UNSUPPORTED, "sub-pixel factor %d needs c_out %% r^2 == 0 and an output tile (%d "
                                              "channels) of whole 16-channel groups per sub-pixel", a.d2s, a.n_t);
    }
    a.num_kb = g.k_pad / 64;
    a.cin_kb = g.cin_pad / 64;
    a.half = g.half;
    a.cin_h = g.cin_pad / 32;
    a.gather = g.gather;
    // exact fp32 chunks: 1024 products of |x| <= 127 (INT8 codes), 512 of |x| <= 255 (centred affine codes)
    a.affine = L->in_affine ? 1 : 0;
    a.a_f16 = L->in_f16 ? 1 : 0;
    a.out_f16 = L->out_f16 ? 1 : 0;
    if (a.a_f16 && (g.gather || g.half || a.affine))
        return fail(HATQ_ERR_UNSUPPORTED, "an fp16 operand needs c_in %% 64 == 0 or 16 or 48, and INT8 codes");
    if (a.out_f16 && (L->out_f32 || (og && og->d2s)))
        return fail(HATQ_ERR_UNSUPPORTED, "fp16 code output needs INT8 output without the sub-pixel rearrangement");
    a.chunk_kb = a.affine ? 8 : 16;
    a.b_bytes = a.n_t * 128;
    a.raw_bytes = g.gather ? 0 : ((a.affine || a.a_f16) ? 16384 : 8192);
    a.n_tiles_n = d->c_out / a.n_t;
    {
        const long long nt = (long long)n * a.tiles_w * a.tiles_h * a.n_tiles_n;
        if (nt >= (1LL << 31)) return fail(HATQ_ERR_UNSUPPORTED, "too many output tiles");
        a.num_tiles = (int)nt;
    }
    // TMEM (all 512 columns): two fp32 regions of n_t columns, exact chunk g
    // of the reduction accumulating in region g & 1, then the ring of fp16
    // A-operand slots. Without drains the two epilogue warpgroups alternate
    // tiles (nbuf = 2); with drains both take every chunk, each for half of
    // the columns, keeping int32 partials in registers (nbuf = 1). A
    // 128-column transform group (n_t = 128) is always shared by both
    // warpgroups, one half each (nbuf = 1).
    const bool drains = a.num_kb > a.chunk_kb;
    a.buf_cols = a.n_t;
    a.nbuf = (drains || g.G == 128) ? 1 : 2;
    a.tmem_cols = 512;
    a.a_col = 2 * a.n_t;
    a.seg = g.seg;
    // shared memory: [stages][output tiles][barriers | gather table | constants | window]
    const int esz = L->out_f32 ? 4 : 1;
    a.row_stride = a.n_t * esz + 16;                 // padded rows: 8 consecutive rows hit 8 bank groups
    a.staging_bytes = L->out_f32 ? 0 : a.nbuf * kTileRows * a.row_stride;   // float32 output is stored directly
    a.win_h = (a.th - 1) * d->stride + d->kh;
    a.win_w = (a.tw - 1) * d->stride + d->kw;
    a.win_pitch = a.win_tma ? window_box_bytes(a.tw, d->stride, d->kw, d->c_in) : (a.win_w * d->c_in + 15) & ~15;
    a.win_tma_bytes = a.win_tma ? a.win_pitch * a.win_h : 0;
    a.win_buf = (a.win_h * a.win_pitch + 16 + 127) & ~127;  // + 16: the gather reads up to 11 bytes past a segment
    // + 16 bytes: the gather reads up to 11 bytes past a row segment
    const int win_bytes = g.gather ? a.win_buf * (a.win_tma ? 2 : 1) : 0;
    const int table_bytes = g.gather ? a.num_kb * 8 * 4 : 0;
    const bool general = L->act == HATQ_ACT_SILU || L->act == HATQ_ACT_GELU;
    const int const_bytes = ((4 * d->c_out * 4 + 127) & ~127) + (general ? 256 : 0);
    const int fixed = 1024 /* align */ + 8 * (3 * 8 + 13) + 16 + 128 + table_bytes + const_bytes + win_bytes;
    const int budget = 227 * 1024 - 1024 /* static */ - fixed - a.staging_bytes;
    // a stage holds `sub` 64-wide reduction blocks: [weights x sub | INT8 box x sub].
    // The cost of a stage is dominated by its barrier hand-offs, not its bytes,
    // so take the widest stage that still leaves two stages and two A slots:
    // four blocks (two 4-block stages, 2 x 128 TMEM columns), else two (three
    // stages, 2 x 64 columns), else one.
    const int one = a.b_bytes + a.raw_bytes;
    const int free_cols = 512 - a.a_col;
    a.sub = 1;
    if (!g.gather && a.num_kb >= 4 && budget / (4 * one) >= 2 && free_cols >= 256) a.sub = 4;
    else if (!g.gather && a.num_kb > 1 && budget / (2 * one) >= 3 && free_cols >= 128) a.sub = 2;
    a.a_slots = free_cols / (32 * a.sub);
    if (a.a_slots > 4) a.a_slots = 4;
    if (a.a_slots < 2) return fail(HATQ_ERR_UNSUPPORTED, "no TMEM room for the A operand (n_t=%d)", a.n_t);
    a.stage_bytes = a.sub * one;
    a.b_off = 0;
    a.raw_off = a.sub * a.b_bytes;
    a.stages = budget / a.stage_bytes;
    if (a.stages > 8) a.stages = 8;
    if (g.gather && a.stages > 4) a.stages = 4;
    if (a.stages < 2) return fail(HATQ_ERR_UNSUPPORTED, "tile does not fit in shared memory");
    const int bar_bytes = 8 * (3 * a.stages + 13) + 16;
    a.const_off = (bar_bytes + table_bytes + 127) & ~127;
    a.win_off = a.const_off + const_bytes;
    const int smem_bytes = a.stages * a.stage_bytes + a.staging_bytes + 1024 + a.win_off + win_bytes;
    // the exchange of a 128-wide next-layer transform uses the output tile: 2 x 128 rows x 64 bytes
    if (g.G == 128 && L->hb_next == 128 && a.staging_bytes < 2 * kTileRows * 64)
        return fail(HATQ_ERR_UNSUPPORTED, "output tile too small for the 128-wide transition exchange");
    if (smem_bytes > 227 * 1024 - 1024) return fail(HATQ_ERR_UNSUPPORTED, "shared memory budget exceeded (%d bytes)", smem_bytes);
    if (a.affine && g.gather) return fail(HATQ_ERR_UNSUPPORTED, "affine activations need c_in % 16 == 0");
    a.x = static_cast<const int8_t *>(x);
    a.b_int = L->b_int;
    a.mult = L->mult;
    a.deq = L->deq;
    a.s_w = L->s_w;
    a.affine_s = affine_s;
    a.inv_gamma = d->form == HATQ_WH ? (float)(1.0 / std::sqrt((double)d->hb_out)) : 1.0f;
    a.shift = L->shift;
    a.hb_out = d->form == HATQ_WH ? d->hb_out : 0;
    a.hb_next = L->hb_next;
    a.act = L->act == HATQ_ACT_RELU ? 1 : 0;
    a.general = general ? 1 : 0;
    a.shift_in = L->shift_in;
    a.mult_in = L->mult_in;
    a.lut_off = a.const_off + ((4 * d->c_out * 4 + 127) & ~127);
    std::memcpy(a.lut, L->lut, sizeof a.lut);
    a.out_f32 = L->out_f32;
    a.y = y;
    a.err = err_word();
    if (!a.err) return fail(HATQ_ERR_CUDA, "no CUDA device");

    CUtensorMap tmB, tmA;
    std::memcpy(&tmB, L->opaque, sizeof tmB);
    if (!g.gather) {
        EncodeTiledFn enc = encode_fn();
        if (!enc) return fail(HATQ_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
        // INT8 codes (64-byte box rows, 64-byte swizzle), or centred int16 affine codes / fp16
        // operand codes (128-byte rows, 128-byte swizzle); 32-channel boxes take half the row and
        // the swizzle of that width
        const bool wide = a.affine || a.a_f16;
        const cuuint64_t es = wide ? 2 : 1;
        const cuuint64_t dims[4] = {(cuuint64_t)d->c_in, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)n};
        const cuuint64_t strides[3] = {(cuuint64_t)d->c_in * es, (cuuint64_t)w * d->c_in * es,
                                       (cuuint64_t)h * w * d->c_in * es};
        // c_in % 64 == 32: 32-channel boxes (32- or 64-byte rows, swizzled to match), two per block
        const cuuint32_t box[4] = {g.half ? 32u : 64u, (cuuint32_t)(a.tw * d->stride), (cuuint32_t)(a.th * d->stride), 1};
        const cuuint32_t estr[4] = {1, (cuuint32_t)d->stride, (cuuint32_t)d->stride, 1};
        CUresult r = enc(&tmA, wide ? CU_TENSOR_MAP_DATA_TYPE_UINT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 4,
                         const_cast<void *>(x), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         g.half ? (wide ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B)
                                : (wide ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B),
                         CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return fail(HATQ_ERR_CUDA, "activation tensor map encoding failed (%d)", (int)r);
    } else if (a.win_tma) {
        // the input as a [n][h][w c] byte tensor; one box = one tile's window rows
        EncodeTiledFn enc = encode_fn();
        if (!enc) return fail(HATQ_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
        const cuuint64_t dims[3] = {(cuuint64_t)w * d->c_in, (cuuint64_t)h, (cuuint64_t)n};
        const cuuint64_t strides[2] = {(cuuint64_t)w * d->c_in, (cuuint64_t)h * w * d->c_in};
        const cuuint32_t box[3] = {(cuuint32_t)a.win_pitch, (cuuint32_t)a.win_h, 1};
        const cuuint32_t estr[3] = {1, 1, 1};
        CUresult r = enc(&tmA, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void *>(x), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return fail(HATQ_ERR_CUDA, "input window tensor map encoding failed (%d)", (int)r);
    } else {
        tmA = tmB;
    }
    cudaError_t e = hatq::launch_conv(tmA, tmB, a, smem_bytes, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "convolution launch");
    return HATQ_OK;
}

// Output parity class p of a transposed convolution (kernel k, stride s,
// padding pad): its taps are ky = p + pad (mod s); sub-convolution tap j is
// kernel tap ky_max - s j and reads input row r + j - off for class pixel r,
// with off = (ky_max - p - pad) / s.
struct TClass {
    int taps, ky_max, off;
};

TClass transposed_class(int k, int s, int pad, int p) {
    for (int ky = k - 1; ky >= 0; --ky)
        if (((ky - p - pad) % s + s) % s == 0) return TClass{ky / s + 1, ky, (ky - p - pad) / s};
    return TClass{0, 0, 0};
}

hatq_status transposed_sub_desc(const hatq_conv_desc *d, int cls, hatq_conv_desc *sub, TClass *ty, TClass *tx) {
    hatq_status st = check_desc(d);
    if (st != HATQ_OK) return st;
    if (d->form == HATQ_TRANSFORM || (d->form == HATQ_DH && !pow2(d->hb_in)))
        return fail(HATQ_ERR_UNSUPPORTED, "transposed convolutions take DH / WH layers with block transforms");
    const int s = d->stride;
    if (d->kh < s || d->kw < s) return fail(HATQ_ERR_UNSUPPORTED, "a transposed convolution needs kh, kw >= stride");
    if (cls < 0 || cls >= s * s) return fail(HATQ_ERR_INVALID_ARG, "class %d out of range for stride %d", cls, s);
    *ty = transposed_class(d->kh, s, d->pad, cls / s);
    *tx = transposed_class(d->kw, s, d->pad, cls % s);
    *sub = *d;
    sub->kh = ty->taps;
    sub->kw = tx->taps;
    sub->stride = 1;
    sub->pad = 0;
    return HATQ_OK;
}

// phi_int parameters of GDN / IGDN (the rules of hatq_prepare_gdn_host).
struct GdnHost {
    std::vector<int32_t> G, B;
    int e = 0, t = 0, shift_in = 0;
    long long P = 0, d_max = 0, mult_in = 0;
};

hatq_status gdn_host(int c, const double *beta, const double *gamma, float s_z, float s_u, int inverse, float s_y,
                     int hb_next, GdnHost &h) {
    if (!beta || !gamma) return fail(HATQ_ERR_INVALID_ARG, "null beta or gamma");
    if (c != 64 && c != 128 && c != 192 && c != 256) return fail(HATQ_ERR_UNSUPPORTED, "GDN channels must be 64, 128, 192 or 256");
    if (hb_next != 0 && (!pow2(hb_next) || hb_next > 64))
        return fail(HATQ_ERR_UNSUPPORTED, "hb_next must be 0 or a power of two <= 64");
    if (!(s_z > 0.f) || !(s_u > 0.f) || !(s_y > 0.f) || !std::isfinite(s_z) || !std::isfinite(s_u) || !std::isfinite(s_y))
        return fail(HATQ_ERR_INVALID_ARG, "scales must be positive and finite");
    const size_t cc = (size_t)c * c;
    const double sz = (double)s_z, su = (double)s_u, sy = (double)s_y;
    std::vector<double> gs(cc);
    double gmax = 0.0, bmax = 0.0;
    for (int i = 0; i < c; ++i) {
        if (!(beta[i] > 0.0) || !std::isfinite(beta[i])) return fail(HATQ_ERR_INVALID_ARG, "beta must be positive and finite");
        bmax = std::max(bmax, beta[i]);
    }
    for (size_t i = 0; i < cc; ++i) {
        if (!(gamma[i] >= 0.0) || !std::isfinite(gamma[i])) return fail(HATQ_ERR_INVALID_ARG, "gamma must be >= 0 and finite");
        gs[i] = gamma[i] * sz * sz;
        gmax = std::max(gmax, gs[i]);
    }
    h.G.assign(cc, 0);
    h.B.assign(c, 0);
    bool found = false;
    for (int e = 62; e >= -125 && !found; --e) {
        const double sc = std::ldexp(1.0, e);
        if (gmax * sc >= 511.5 || bmax * sc >= 2147483648.0) continue;
        long long dmax = 0;
        for (int i = 0; i < c; ++i) {
            const double b = std::nearbyint(beta[i] * sc);
            h.B[i] = (int32_t)(b < 1.0 ? 1.0 : b);
            long long sum = 0;
            for (int j = 0; j < c; ++j) {
                h.G[(size_t)i * c + j] = (int32_t)std::nearbyint(gs[(size_t)i * c + j] * sc);
                sum += h.G[(size_t)i * c + j];
            }
            dmax = std::max(dmax, (long long)h.B[i] + 16129LL * sum);
        }
        if (dmax < (1LL << 31)) {
            h.e = e;
            h.d_max = dmax;
            found = true;
        }
    }
    if (!found) return fail(HATQ_ERR_OVERFLOW, "no scaling keeps the GDN pool in range");
    const double q = sz / su;
    const double r2 = q * q * std::ldexp(1.0, inverse ? -h.e : h.e);
    typedef unsigned __int128 u128;
    const u128 lim = (u128)1 << 63;
    found = false;
    for (int t = 62; t >= 0 && !found; --t) {
        const double pv = std::nearbyint(std::ldexp(r2, t));
        if (pv >= 4611686018427387904.0) continue;          // 4 P 127^2 would pass 2^63
        const long long P = (long long)pv;
        bool ok;
        if (inverse)
            ok = (u128)64009 << t < lim && (u128)4 * (u128)P * 16129u * (u128)h.d_max < lim;
        else
            ok = ((u128)64009 * (u128)h.d_max) << t < lim && (u128)4 * (u128)P * 16129u < lim;
        if (ok) {
            h.P = P;
            h.t = t;
            found = true;
        }
    }
    if (!found) return fail(HATQ_ERR_OVERFLOW, "no fixed-point R^2 fits the 63-bit tests");
    if (h.P < (1LL << 15)) return fail(HATQ_ERR_OVERFLOW, "fewer than 16 bits in the fixed-point R^2");
    // Eq. supp_general_input_scale: s_u / (gamma_in,next s_y)
    const double g_in = hb_next ? std::sqrt((double)hb_next) : 1.0;
    std::vector<int32_t> m_in;
    hatq_status st = fixed_point({su / (g_in * sy)}, {127LL}, hb_next ? hb_next : 1, m_in, h.shift_in);
    if (st != HATQ_OK) return st;
    h.mult_in = m_in[0];
    return HATQ_OK;
}

}  // namespace

extern "C" {

hatq_status hatq_conv2d_i8(const int8_t *x, int n, int h, int w, const hatq_prepared *L, void *y, hatq_stream stream) {
    return conv_launch(x, n, h, w, L, y, stream, nullptr);
}

hatq_status hatq_conv2d_i8_subpixel(const int8_t *x, int n, int h, int w, const hatq_prepared *L, int r, void *y,
                                    hatq_stream stream) {
    if (!L) return fail(HATQ_ERR_INVALID_ARG, "null layer");
    if (r < 2 || r > 4) return fail(HATQ_ERR_INVALID_ARG, "sub-pixel factor must be 2..4");
    const hatq_conv_desc *d = &L->d;
    if (h < 1 || w < 1) return fail(HATQ_ERR_INVALID_ARG, "bad input shape");
    const int ho = (h + 2 * d->pad - d->kh) / d->stride + 1, wo = (w + 2 * d->pad - d->kw) / d->stride + 1;
    if (h + 2 * d->pad < d->kh || w + 2 * d->pad < d->kw || ho < 1 || wo < 1)
        return fail(HATQ_ERR_INVALID_ARG, "input smaller than the kernel");
    const OutGrid og{d->pad, d->pad, ho, wo, ho, wo, 1, 0, 0, r};
    return conv_launch(x, n, h, w, L, y, stream, &og);
}

hatq_status hatq_prepare_weights_affine(const hatq_conv_desc *d, const float *w_ohwi, const float *bias, int act,
                                        hatq_prepared *out, hatq_stream stream) {
    hatq_conv_desc dop;
    hatq_status st = operand_desc(d, 0, &dop);
    if (st != HATQ_OK) return st;
    if (act != HATQ_ACT_NONE && act != HATQ_ACT_RELU)
        return fail(HATQ_ERR_UNSUPPORTED, "affine layers take no activation or ReLU");
    if (d->c_in % 16) return fail(HATQ_ERR_UNSUPPORTED, "affine activations need c_in % 16 == 0");
    Geometry g;
    if ((st = validate_prepare(&dop, w_ohwi, 1.f, 1.f, act, 0, 1, &g)) != HATQ_OK) return st;
    if ((st = check_out_buffers(out)) != HATQ_OK) return st;
    HostLayer hl(dop.c_out, g.k_pad);
    std::vector<double> bbar(dop.c_out);
    st = prepare_core(d, w_ohwi, bias, 1.f, 1.f, act, 0, 1, nullptr, 0, hl.w_i8.data(), hl.w_f16.data(), hl.b_int.data(),
                      hl.mult.data(), hl.deq.data(), hl.s_w.data(), &hl.shift, bbar.data());
    if (st != HATQ_OK) return st;
    // the bias stays real-valued (the activation scale is per input): beta_c = b_bar_c / gamma_out
    const double g_out = d->form == HATQ_WH ? std::sqrt((double)d->hb_out) : 1.0;
    for (int o = 0; o < dop.c_out; ++o) {
        hl.b_int[o] = 0;
        hl.mult[o] = 0;
        hl.deq[o] = (float)(bbar[o] / g_out);
    }
    if ((st = upload_layer(dop, g, hl, act, 0, 1, 1.f, 0.f, nullptr, out, stream)) != HATQ_OK) return st;
    out->in_affine = 1;
    out->s_x = 0.f;
    return HATQ_OK;
}

hatq_status hatq_quantize_act_affine(const void *x, int n, int h, int w, int c, int hb, int16_t *y, float *params,
                                     void *workspace, hatq_stream stream) {
    if (n == 0 && h >= 0 && w >= 0 && c >= 0) return HATQ_OK;
    if (!x || !y || !params || !workspace) return fail(HATQ_ERR_INVALID_ARG, "null argument");
    if (!aligned16(x) || !aligned16(y) || !aligned16(workspace))
        return fail(HATQ_ERR_INVALID_ARG, "input, output and workspace must be 16-byte aligned");
    if (n < 0 || h < 0 || w < 0 || c < 16 || c % 16) return fail(HATQ_ERR_INVALID_ARG, "shape must be n,h,w >= 0, c % 16 == 0");
    if (!pow2(hb) || hb > 256 || c % hb) return fail(HATQ_ERR_INVALID_ARG, "hb must be a power of two <= 256 dividing c");
    const long long total = (long long)n * h * w * c;
    if (total == 0) return HATQ_OK;
    hatq::AffineQuantArgs a{};
    a.x = x;
    a.y = y;
    a.total = total;
    a.hb = hb;
    a.p = static_cast<hatq::AffineParams *>(workspace);
    a.params_out = params;
    cudaError_t e = hatq::launch_act_affine(a, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "affine quantization launch");
    return HATQ_OK;
}

hatq_status hatq_conv2d_affine(const int16_t *x, int n, int h, int w, const hatq_prepared *L, const float *params,
                               float *y, hatq_stream stream) {
    if (!params) return fail(HATQ_ERR_INVALID_ARG, "null scale");
    return conv_launch(x, n, h, w, L, y, stream, nullptr, params);
}

hatq_status hatq_transposed_sizes(const hatq_conv_desc *d, int cls, size_t *w_elems, size_t *ch_elems) {
    hatq_conv_desc sub;
    TClass ty, tx;
    hatq_status st = transposed_sub_desc(d, cls, &sub, &ty, &tx);
    if (st != HATQ_OK) return st;
    return hatq_prepared_sizes(&sub, w_elems, ch_elems);
}

hatq_status hatq_prepare_weights_transposed(const hatq_conv_desc *d, int out_pad, const float *w_ohwi, const float *bias,
                                            float s_x, float s_y, int act, int hb_next, int out_f32,
                                            hatq_prepared_transposed *out, hatq_stream stream) {
    if (!out) return fail(HATQ_ERR_INVALID_ARG, "null output struct");
    hatq_conv_desc sub0;
    TClass ty, tx;
    hatq_status st = transposed_sub_desc(d, 0, &sub0, &ty, &tx);
    if (st != HATQ_OK) return st;
    const int s = d->stride;
    if (out_pad < 0 || out_pad >= s) return fail(HATQ_ERR_INVALID_ARG, "output padding must be in [0, stride)");
    if (act == HATQ_ACT_SILU || act == HATQ_ACT_GELU)
        return fail(HATQ_ERR_UNSUPPORTED, "transposed layers take the homogeneous transition (none / ReLU)");
    Geometry gf;
    if ((st = validate_prepare(d, w_ohwi, s_x, s_y, act, hb_next, out_f32, &gf)) != HATQ_OK) return st;
    for (int c = 0; c < s * s; ++c)
        if ((st = check_out_buffers(&out->sub[c])) != HATQ_OK) return st;
    // the whole kernel, transformed and quantized once
    HostLayer full(d->c_out, gf.k_pad);
    st = prepare_core(d, w_ohwi, bias, s_x, s_y, act, hb_next, out_f32, nullptr, 0, full.w_i8.data(), full.w_f16.data(),
                      full.b_int.data(), full.mult.data(), full.deq.data(), full.s_w.data(), &full.shift);
    if (st != HATQ_OK) return st;
    const int ci = d->c_in, co = d->c_out;
    auto full_index = [&](int ky, int kx, int c) -> long long {
        return gf.gather ? (long long)ky * gf.seg + (long long)kx * ci + c : (long long)(ky * d->kw + kx) * gf.cin_pad + c;
    };
    for (int cls = 0; cls < s * s; ++cls) {
        hatq_conv_desc sub;
        if ((st = transposed_sub_desc(d, cls, &sub, &ty, &tx)) != HATQ_OK) return st;
        Geometry gs;
        if ((st = geometry(&sub, hb_next, &gs)) != HATQ_OK) return st;
        HostLayer hs(co, gs.k_pad);
        hs.b_int = full.b_int;
        hs.mult = full.mult;
        hs.deq = full.deq;
        hs.s_w = full.s_w;
        hs.shift = full.shift;
        for (size_t k = 0; k < hs.w_f16.size(); ++k) hs.w_f16[k] = f16_bits(0);
        for (int o = 0; o < co; ++o)
            for (int j = 0; j < ty.taps; ++j)
                for (int l = 0; l < tx.taps; ++l)
                    for (int c = 0; c < ci; ++c) {
                        const long long src = (long long)o * gf.k_pad + full_index(ty.ky_max - s * j, tx.ky_max - s * l, c);
                        const long long dst = (long long)o * gs.k_pad +
                                              (gs.gather ? (long long)j * gs.seg + (long long)l * ci + c
                                                         : (long long)(j * tx.taps + l) * gs.cin_pad + c);
                        hs.w_i8[dst] = full.w_i8[src];
                        hs.w_f16[dst] = full.w_f16[src];
                    }
        if ((st = upload_layer(sub, gs, hs, act, hb_next, out_f32, s_x, s_y, nullptr, &out->sub[cls], stream)) != HATQ_OK)
            return st;
        out->pad_y[cls] = ty.off;
        out->pad_x[cls] = tx.off;
    }
    out->d = *d;
    out->out_pad = out_pad;
    out->classes = s * s;
    return HATQ_OK;
}

hatq_status hatq_conv_transpose2d_i8(const int8_t *x, int n, int h, int w, const hatq_prepared_transposed *T, void *y,
                                     hatq_stream stream) {
    if (!T) return fail(HATQ_ERR_INVALID_ARG, "null layer");
    const int s = T->d.stride;
    if (s < 1 || s > 2 || T->classes != s * s) return fail(HATQ_ERR_INVALID_ARG, "transposed layer is not prepared");
    if (h < 1 || w < 1 || n < 0) return fail(HATQ_ERR_INVALID_ARG, "bad input shape");
    const int ho = (h - 1) * s - 2 * T->d.pad + T->d.kh + T->out_pad;
    const int wo = (w - 1) * s - 2 * T->d.pad + T->d.kw + T->out_pad;
    if (ho < 1 || wo < 1) return fail(HATQ_ERR_INVALID_ARG, "empty output");
    for (int cls = 0; cls < s * s; ++cls) {
        const int py = cls / s, px = cls % s;
        const int hc = ho > py ? (ho - py + s - 1) / s : 0, wc = wo > px ? (wo - px + s - 1) / s : 0;
        if (!hc || !wc) continue;
        const OutGrid og{T->pad_y[cls], T->pad_x[cls], hc, wc, ho, wo, s, py, px, 0};
        hatq_status st = conv_launch(x, n, h, w, &T->sub[cls], y, stream, &og);
        if (st != HATQ_OK) return st;
    }
    return HATQ_OK;
}

int hatq_layer_launches(int x_kind, float s_in, const hatq_prepared *L) {
    if (!L) return -1;
    if (x_kind == HATQ_IN_OPERAND) return 1;
    if (L->in_f16) return -1;
    if (L->d.form == HATQ_TRANSFORM) return x_kind == HATQ_IN_I8 ? 1 : -1;
    if (L->d.form == HATQ_DH && !pow2(L->d.hb_in)) return -1;   // paper order: operand from the transform layer
    if (x_kind == HATQ_IN_I8) return (L->d.form == HATQ_WH && s_in == L->s_x) ? 1 : 2;
    if (x_kind == HATQ_IN_F16) return 2;
    return -1;
}

hatq_status hatq_layer(const void *x, int x_kind, float s_in, int n, int h, int w, const hatq_prepared *L, void *y,
                       void *scratch, size_t scratch_bytes, hatq_stream stream) {
    if (!L) return fail(HATQ_ERR_INVALID_ARG, "null layer");
    if (n == 0 && h >= 1 && w >= 1) return HATQ_OK;                    // empty batch: nothing to do
    if (!x || !y) return fail(HATQ_ERR_INVALID_ARG, "null argument");
    const hatq_conv_desc *d = &L->d;
    if (L->in_f16 && x_kind != HATQ_IN_OPERAND)
        return fail(HATQ_ERR_UNSUPPORTED, "a layer with an fp16 operand takes it as HATQ_IN_OPERAND");
    if (x_kind == HATQ_IN_OPERAND || (x_kind == HATQ_IN_I8 && d->form == HATQ_WH && s_in == L->s_x) ||
        (x_kind == HATQ_IN_I8 && d->form == HATQ_TRANSFORM))
        return hatq_conv2d_i8(static_cast<const int8_t *>(x), n, h, w, L, y, stream);
    if (x_kind != HATQ_IN_I8 && x_kind != HATQ_IN_F16) return fail(HATQ_ERR_INVALID_ARG, "unknown input kind %d", x_kind);
    if (d->form == HATQ_TRANSFORM) return fail(HATQ_ERR_INVALID_ARG, "a transform layer takes INT8 codes");
    if (d->form == HATQ_DH && !pow2(d->hb_in))
        return fail(HATQ_ERR_UNSUPPORTED, "a paper-order layer consumes the output of its transform layer "
                                          "(hatq_prepare_order_transform) as HATQ_IN_OPERAND");
    const size_t need = (size_t)n * h * w * d->c_in;
    if (!scratch || scratch_bytes < need) return fail(HATQ_ERR_INVALID_ARG, "scratch must hold %zu bytes", need);
    if (d->c_in % 16) return fail(HATQ_ERR_UNSUPPORTED, "an input transform needs c_in % 16 == 0");
    const int hb = d->form == HATQ_DH ? d->hb_in : 1;
    hatq_status st = hatq_quantize_act(x, x_kind, s_in, n, h, w, d->c_in, hb, L->s_x, static_cast<int8_t *>(scratch),
                                       nullptr, nullptr, stream);
    if (st != HATQ_OK) return st;
    return hatq_conv2d_i8(static_cast<const int8_t *>(scratch), n, h, w, L, y, stream);
}

hatq_status hatq_profile_range(const int8_t *x, int n, int h, int w, int c, int hb, int32_t *maxima, uint8_t *expands,
                               hatq_stream stream) {
    if (n < 0 || h < 1 || w < 1 || c < 1) return fail(HATQ_ERR_INVALID_ARG, "bad shape");
    if (!pow2(hb) || hb < 2 || hb > 256 || c % hb)
        return fail(HATQ_ERR_INVALID_ARG, "hb must be a power of two in 2..256 dividing c");
    if (c % 16) return fail(HATQ_ERR_UNSUPPORTED, "profiling needs c % 16 == 0");
    if (n == 0) return HATQ_OK;
    if (!x || !maxima) return fail(HATQ_ERR_INVALID_ARG, "null argument");
    if (reinterpret_cast<uintptr_t>(x) % 16) return fail(HATQ_ERR_INVALID_ARG, "x must be 16-byte aligned");
    const long long per = (long long)h * w * c;
    if (per >= (1LL << 40)) return fail(HATQ_ERR_UNSUPPORTED, "image too large");
    hatq::ProfileArgs a{};
    a.x = x;
    a.per_image = per;
    a.n = n;
    a.hb = hb;
    a.maxima = maxima;
    cudaError_t e = hatq::launch_profile(a, expands, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "profiling launch");
    return HATQ_OK;
}

hatq_status hatq_select_form(const uint8_t *expands, int n, int tau_num, int tau_den, int *form, int *expanded) {
    if (!expands || !form) return fail(HATQ_ERR_INVALID_ARG, "null argument");
    if (n < 1) return fail(HATQ_ERR_INVALID_ARG, "at least one profiled image is required");
    if (tau_den < 1 || tau_num < 0 || tau_num > tau_den)
        return fail(HATQ_ERR_INVALID_ARG, "tau_sel must be a fraction in [0, 1] with a positive denominator");
    long long count = 0;
    for (int k = 0; k < n; ++k) count += expands[k] != 0;
    // p_l = count / n > tau_num / tau_den, cross-multiplied (no rounding)
    *form = count * (long long)tau_den > (long long)n * tau_num ? HATQ_WH : HATQ_DH;
    if (expanded) *expanded = (int)count;
    return HATQ_OK;
}

hatq_status hatq_prepare_gdn_host(int c, const double *beta, const double *gamma, float s_z, float s_u, int inverse,
                                  float s_y, int hb_next, int32_t *g_out, int32_t *b_out, int *e_out, long long *p_out,
                                  int *t_out, long long *mult_in_out, int *shift_in_out) {
    if (!g_out || !b_out || !e_out || !p_out || !t_out || !mult_in_out || !shift_in_out)
        return fail(HATQ_ERR_INVALID_ARG, "null output");
    GdnHost h;
    hatq_status st = gdn_host(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next, h);
    if (st != HATQ_OK) return st;
    std::memcpy(g_out, h.G.data(), (size_t)c * c * 4);
    std::memcpy(b_out, h.B.data(), (size_t)c * 4);
    *e_out = h.e;
    *p_out = h.P;
    *t_out = h.t;
    *mult_in_out = h.mult_in;
    *shift_in_out = h.shift_in;
    return HATQ_OK;
}

hatq_status hatq_prepare_gdn(int c, const double *beta, const double *gamma, float s_z, float s_u, int inverse,
                             float s_y, int hb_next, hatq_prepared_gdn *out, hatq_stream stream) {
    if (!out) return fail(HATQ_ERR_INVALID_ARG, "null output struct");
    if (!out->g_f16 || !out->b_pool) return fail(HATQ_ERR_INVALID_ARG, "g_f16 and b_pool must be set before preparation");
    if (!aligned16(out->g_f16) || !aligned16(out->b_pool)) return fail(HATQ_ERR_INVALID_ARG, "device buffers must be 16-byte aligned");
    GdnHost h;
    hatq_status st = gdn_host(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next, h);
    if (st != HATQ_OK) return st;
    std::vector<uint16_t> g16((size_t)c * c);
    for (size_t i = 0; i < g16.size(); ++i) g16[i] = f16_bits(h.G[i]);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e;
    if ((e = cudaMemcpyAsync(out->g_f16, g16.data(), g16.size() * 2, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out->b_pool, h.B.data(), (size_t)c * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaStreamSynchronize(s)) != cudaSuccess)
        return cuda_fail(e, "upload of GDN parameters");
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(HATQ_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    // G: [c][c] fp16 (K innermost), 64 x c box, 128-byte swizzle
    CUtensorMap tm;
    const cuuint64_t dims[2] = {(cuuint64_t)c, (cuuint64_t)c};
    const cuuint64_t strides[1] = {(cuuint64_t)c * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)c};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, out->g_f16, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HATQ_ERR_CUDA, "pool tensor map encoding failed (%d)", (int)r);
    std::memcpy(out->opaque, &tm, sizeof tm);
    out->c = c;
    out->inverse = inverse ? 1 : 0;
    out->hb_next = hb_next;
    out->e = h.e;
    out->t = h.t;
    out->shift_in = h.shift_in;
    out->P = h.P;
    out->mult_in = h.mult_in;
    out->s_z = s_z;
    out->s_u = s_u;
    out->s_y = s_y;
    return HATQ_OK;
}

hatq_status hatq_gdn(const int8_t *z, int n, int h, int w, const hatq_prepared_gdn *g, int8_t *y, hatq_stream stream) {
    if (!g) return fail(HATQ_ERR_INVALID_ARG, "null prepared GDN");
    if (n < 0 || h < 0 || w < 0) return fail(HATQ_ERR_INVALID_ARG, "negative shape");
    const int c = g->c;
    if (c != 64 && c != 128 && c != 192 && c != 256) return fail(HATQ_ERR_INVALID_ARG, "the struct was not prepared");
    const long long pixels = (long long)n * h * w;
    if (pixels == 0) return HATQ_OK;
    if (!z || !y) return fail(HATQ_ERR_INVALID_ARG, "null tensor");
    if (!aligned16(z) || !aligned16(y)) return fail(HATQ_ERR_INVALID_ARG, "z and y must be 16-byte aligned");
    if (pixels > (1LL << 31) - 256) return fail(HATQ_ERR_UNSUPPORTED, "at most 2^31 - 256 pixels per call");
    const int8_t *zl = z, *zh = z + pixels * c, *yl = y, *yh = y + pixels * c;
    if (zl < yh && yl < zh) return fail(HATQ_ERR_INVALID_ARG, "z and y overlap");
    int dev = 0, smem_max = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&smem_max, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess)
        return cuda_fail(e, "device query");
    hatq::GdnArgs a{};
    a.z = z;
    a.y = y;
    a.pixels = pixels;
    a.c = c;
    a.inverse = g->inverse;
    a.hb_next = g->hb_next;
    a.t = g->t;
    a.shift_in = g->shift_in;
    a.P = (unsigned long long)g->P;
    a.sr = (float)std::sqrt(std::ldexp((double)g->P, -g->t));
    a.mult_in = g->mult_in;
    a.b_pool = g->b_pool;
    a.err = err_word();
    if (!a.err) return fail(HATQ_ERR_CUDA, "no CUDA device");
    a.num_tiles = (int)((pixels + 127) / 128);
    // shared memory: G, nz z tiles, the u rows, B, barriers (plus the 1024-byte alignment slack)
    const int g_bytes = c * c * 2, z_bytes = 128 * c, u_bytes = 128 * (c + 16);
    auto layout = [&](int nz) {
        a.nz = nz;
        a.z_off = g_bytes;
        a.u_off = a.z_off + nz * z_bytes;
        a.b_off = (a.u_off + u_bytes + 127) & ~127;
        a.lut_off = a.b_off + 8 * c;
        a.bar_off = (a.lut_off + 255 * (g->hb_next > 1 ? g->hb_next : 1) + 1 + 63) & ~63;
        return a.bar_off + 64 + 1024;
    };
    int smem = layout(2);
    if (smem > smem_max) smem = layout(1);
    if (smem > smem_max) return fail(HATQ_ERR_UNSUPPORTED, "the GDN tile does not fit shared memory");
    a.tmem_cols = 512;                   // A limbs (c columns) and two 128-column accumulator buffers
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(HATQ_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    CUtensorMap tmZ, tmG;
    std::memcpy(&tmG, g->opaque, sizeof tmG);
    const cuuint64_t dims[2] = {(cuuint64_t)c, (cuuint64_t)pixels};
    const cuuint64_t strides[1] = {(cuuint64_t)c};
    const cuuint32_t box[2] = {64, 128};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&tmZ, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t *>(z), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HATQ_ERR_CUDA, "preactivation tensor map encoding failed (%d)", (int)r);
    if ((e = hatq::launch_gdn(tmZ, tmG, a, smem, reinterpret_cast<cudaStream_t>(stream))) != cudaSuccess)
        return cuda_fail(e, "GDN launch");
    return HATQ_OK;
}

hatq_status hatq_set_operand_format(hatq_prepared *L, int in_f16, int out_f16) {
    if (!L) return fail(HATQ_ERR_INVALID_ARG, "null layer");
    if ((in_f16 != 0 && in_f16 != 1) || (out_f16 != 0 && out_f16 != 1))
        return fail(HATQ_ERR_INVALID_ARG, "in_f16 and out_f16 must be 0 or 1");
    // the fp16 tile is read by the MMAs in place as whole 64-channel rows, which a layer whose taps
    // are packed at 32-channel granularity (c_in % 64 == 32) does not have
    if (in_f16 && (L->gather || L->in_affine || L->d.form == HATQ_TRANSFORM || L->d.c_in % 64 == 32))
        return fail(HATQ_ERR_UNSUPPORTED, "an fp16 operand needs an INT8 convolution with c_in %% 16 == 0 and "
                                          "c_in %% 64 != 32");
    if (out_f16 && L->out_f32) return fail(HATQ_ERR_UNSUPPORTED, "fp16 code output needs INT8 output");
    L->in_f16 = in_f16;
    L->out_f16 = out_f16;
    return HATQ_OK;
}

hatq_status hatq_selftest_wait(unsigned long long limit_cycles, hatq_stream stream) {
    if (limit_cycles == 0 || limit_cycles > 4000000000ull) return fail(HATQ_ERR_INVALID_ARG, "limit must be in 1..4e9 cycles");
    int *p = err_word();
    if (!p) return fail(HATQ_ERR_CUDA, "no CUDA device");
    cudaError_t e = hatq::launch_wait_selftest(p, (long long)limit_cycles, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "self-test launch");
    return HATQ_OK;
}

hatq_status hatq_sync_status(hatq_stream stream) {
    cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronization");
    int *p = err_word();
    if (!p) return fail(HATQ_ERR_CUDA, "no CUDA device");
    int v = 0;
    if ((e = cudaMemcpy(&v, p, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(e, "error word read");
    if (v != 0) {
        const int zero = 0;
        cudaMemcpy(p, &zero, sizeof zero, cudaMemcpyHostToDevice);
        if (v == hatq::kErrWaitTimeout) return fail(HATQ_ERR_TIMEOUT, "a device-side bounded wait expired");
        return fail(HATQ_ERR_OVERFLOW, "a device-side bound check failed (code %d)", v);
    }
    return HATQ_OK;
}

}  // extern "C"
