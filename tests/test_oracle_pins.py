"""Pins for the CPU oracle: each check compares the oracle with something
other than itself (a closed form, an identity of the paper, a worked table,
brute force, exact rational arithmetic)."""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import hatq_oracle as O
from synth import inputs as I

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def popcount_sign(m):
    """Closed form of the Sylvester matrix: H~[i][j] = (-1)^popcount(i & j)."""
    i = np.arange(m)[:, None]
    j = np.arange(m)[None, :]
    pc = np.vectorize(lambda v: bin(int(v)).count("1"))(i & j)
    return np.where(pc % 2 == 0, 1, -1)


# ---------------------------------------------------------------- Hadamard (T1)

@pytest.mark.parametrize("m", [1, 2, 4, 8, 16, 32, 64, 128, 256])
def test_sylvester_orthogonal_closed_form(m):
    H = O.sylvester(m)
    assert np.array_equal(H @ H.T, m * np.eye(m, dtype=np.int64))          # Eq. supp_hadamard_properties
    assert np.array_equal(H, popcount_sign(m))
    assert np.all(H[0] == 1) and np.all(H[:, 0] == 1)                        # constant basis h0 first
    assert np.array_equal(H, H.T)


def test_sylvester_h4_golden():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "sylvester_h4.txt")) if not l.startswith("#")]
    ref = np.array([[int(v) for v in r] for r in rows if r])
    assert np.array_equal(O.sylvester(4), ref)


def test_sylvester_rejects_non_power_of_two():
    with pytest.raises(ValueError):
        O.sylvester(12)


@pytest.mark.parametrize("c,hb", [(128, 128), (192, 64), (320, 64), (224, 32), (64, 16)])
def test_blockdiag_orthonormal_and_transforms(c, hb):
    T = O.blockdiag_transform(c, hb)
    assert np.allclose(T @ T.T, np.eye(c), atol=1e-13)
    rng = np.random.default_rng(c + hb)
    x = rng.standard_normal((5, c))
    # ordered-loop transform == dense Kronecker matrix product
    assert np.allclose(O.transform_real(x, hb), x @ T, atol=1e-12)
    xi = rng.integers(-127, 128, size=(7, c))
    Hc = np.kron(np.eye(c // hb, dtype=np.int64), popcount_sign(hb))
    assert np.array_equal(O.transform_int(xi, hb), xi @ Hc.T)


def test_parseval():                                                          # T4
    x = I.activations((1, 4, 4, 192), seed=5).astype(np.float64)
    y = O.transform_real(x, 64)
    assert np.allclose(np.sum(y * y), np.sum(x * x), rtol=1e-12)


@pytest.mark.parametrize("hb", [16, 64, 128])
def test_coherent_mean_accumulation(hb):                                      # T3, Eq. hadamard_mean_accumulation
    mu = 0.731
    x = np.full((3, hb), mu)
    y = O.transform_real(x, hb)
    assert np.allclose(y[:, 0], math.sqrt(hb) * mu, rtol=1e-14)
    assert np.allclose(y[:, 1:], 0.0, atol=1e-13)
    yi = O.transform_int(np.full((2, hb), 5), hb)
    assert np.all(yi[:, 0] == 5 * hb) and np.all(yi[:, 1:] == 0)


def test_coherent_mean_general_vector():
    """y0 = C / sqrt(m) * mean(x) for any vector (unpadded: sqrt(C) * mean)."""
    rng = np.random.default_rng(3)
    x = rng.standard_normal((10, 64)) + 2.0
    y = O.transform_real(x, 64)
    assert np.allclose(y[:, 0], math.sqrt(64) * x.mean(axis=1), rtol=1e-12)


# ------------------------------------------------------- function preservation (T2)

def _rel(a, b):
    return float(np.max(np.abs(a - b)) / np.max(np.abs(b)))


@pytest.mark.parametrize("k,stride,pad,c_in,c_out,hb", [(1, 1, 0, 64, 32, 64), (3, 1, 1, 32, 48, 32),
                                                        (5, 2, 2, 64, 16, 16)])
def test_dh_function_preservation(k, stride, pad, c_in, c_out, hb):
    """Eq. hadamard_linear_equivalence: (X H_in)(W H_in)^T = X W^T."""
    x = I.activations((2, 9, 7, c_in), seed=11).astype(np.float64)
    w = I.weights(c_out, k, k, c_in, seed=12).astype(np.float64)
    b = I.bias(c_out, seed=13).astype(np.float64)
    wp, bb = O.transform_weights(w, b, "DH", hb, 0)
    y_ref = O.conv_real(x, w, b, stride, pad)
    y_dh = O.conv_real(O.transform_real(x, hb), wp, bb, stride, pad)
    assert _rel(y_dh, y_ref) < 1e-12


@pytest.mark.parametrize("c_out,hb", [(64, 64), (96, 32), (128, 128)])
def test_wh_function_preservation(c_out, hb):
    """Eq. supp_padded_wh: (X W_bar^T + b_bar) T_out^T = X W^T + b."""
    x = I.activations((1, 6, 6, 16), seed=21).astype(np.float64)
    w = I.weights(c_out, 3, 3, 16, seed=22).astype(np.float64)
    b = I.bias(c_out, seed=23).astype(np.float64)
    wbar, bbar = O.transform_weights(w, b, "WH", 0, hb)
    acc = O.conv_real(x, wbar, bbar, 1, 1)
    y_wh = O.transform_real(acc, hb)
    assert _rel(y_wh, O.conv_real(x, w, b, 1, 1)) < 1e-12
    # and b_bar is b mapped into the output Hadamard basis: b_bar T_out^T = b
    assert np.allclose(O.transform_real(bbar, hb), b, atol=1e-14)


# ------------------------------------------------------------ direct conv (T5)

def im2col_conv(x, w, stride, pad):
    """Independent formulation: explicit patch matrix times weight matrix."""
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    ho = (h + 2 * pad - kh) // stride + 1
    wo = (wd + 2 * pad - kw) // stride + 1
    rows = []
    for b in range(n):
        for oy in range(ho):
            for ox in range(wo):
                patch = []
                for ky in range(kh):
                    for kx in range(kw):
                        iy, ix = oy * stride + ky - pad, ox * stride + kx - pad
                        if 0 <= iy < h and 0 <= ix < wd:
                            patch.extend(int(v) for v in x[b, iy, ix])
                        else:
                            patch.extend([0] * c)
                rows.append(patch)
    A = np.array(rows, dtype=np.int64)
    B = w.reshape(co, -1).astype(np.int64)
    return (A @ B.T).reshape(n, ho, wo, co)


@pytest.mark.parametrize("shape,co,k,stride,pad", [((1, 8, 8, 3), 5, 5, 2, 2), ((2, 7, 5, 16), 8, 3, 1, 1),
                                                   ((1, 6, 6, 32), 4, 1, 1, 0), ((1, 9, 8, 8), 3, 5, 2, 2),
                                                   ((1, 5, 5, 4), 2, 3, 2, 0)])
def test_conv_codes_brute_force(shape, co, k, stride, pad):
    x = I.uniform_codes(shape, seed=31)
    w = I.uniform_codes((co, k, k, shape[3]), seed=32)
    ref = im2col_conv(x, w, stride, pad)
    got = O.conv_codes(x, w, stride, pad)
    assert np.array_equal(got, ref)
    ho, wo = ref.shape[1:3]
    win = O.conv_codes(x, w, stride, pad, window=(1, ho, 0, max(1, wo - 1)))
    assert np.array_equal(win, ref[:, 1:ho, 0:max(1, wo - 1)])
    pix = np.array([[b, oy, ox] for b in range(shape[0]) for oy in range(ho) for ox in range(wo)])
    at = O.conv_codes_at(x, w, stride, pad, pix)
    assert np.array_equal(at, ref.reshape(-1, co))


def test_conv_codes_extreme_values():
    x = np.full((1, 4, 4, 64), -127, dtype=np.int8)
    w = np.full((2, 3, 3, 64), 127, dtype=np.int8)
    acc = O.conv_codes(x, w, 1, 1)
    assert acc[0, 1, 1, 0] == -127 * 127 * 9 * 64
    assert acc[0, 0, 0, 0] == -127 * 127 * 4 * 64


# ------------------------------------------------------- rounding / fixed point (T6)

def test_rshift_rne_matches_exact_rationals():
    rng = np.random.default_rng(7)
    v = np.concatenate([rng.integers(-2 ** 40, 2 ** 40, size=2000),
                        np.array([5, -5, 3, -3, 7, -7, 1, -1, 0, 2 ** 41 + 2 ** 9, -(2 ** 41) - 2 ** 9])])
    for n in [0, 1, 2, 3, 10, 20]:
        got = O.rshift_rne(v, n)
        ref = [O.round_half_even_fraction(Fraction(int(a), 2 ** n)) for a in v]
        assert list(got) == ref


def test_round_half_even_fraction_ties():
    assert [O.round_half_even_fraction(Fraction(k, 2)) for k in (-5, -3, -1, 1, 3, 5)] == [-2, -2, 0, 0, 2, 2]


def test_fixed_point_rule_is_maximal_and_accurate():
    rng = np.random.default_rng(9)
    rho = rng.lognormal(-6, 2, size=64)
    a_bound = rng.integers(10 ** 5, 10 ** 8, size=64)
    for gain in (1, 64, 64 * 64):
        M, n = O.fixed_point(rho, a_bound, gain)
        for r, m in zip(rho, M):
            assert abs(Fraction(int(m)) - Fraction(float(r)) * 2 ** n) <= Fraction(1, 2)
        assert max(M) < 2 ** 31 and max(int(m) * int(a) for m, a in zip(M, a_bound)) * gain < 2 ** 62
        if n < 62:  # n + 1 must violate a bound
            M2 = [int(np.rint(math.ldexp(float(r), n + 1))) for r in rho]
            assert max(M2) >= 2 ** 31 or max(m * int(a) for m, a in zip(M2, a_bound)) * gain >= 2 ** 62


def test_fixed_point_precision_floor():
    with pytest.raises(OverflowError):
        O.fixed_point([1e-9], [2 ** 30], 2 ** 28)


@pytest.mark.parametrize("hb,rho", [(64, 0.5), (64, 0.013), (256, 0.9), (1, 0.37), (16, 3.0)])
def test_activation_multiplier_32bit_bound_and_maximality(hb, rho):
    """Reading R3 for the activation requantizer: the largest n with
    M < 2^31 and M 127 hb < 2^30, so M |y| + 2^(n-1) fits a signed 32-bit word;
    n + 1 breaks the bound; M / 2^n within half a unit of rho 2^n."""
    s_x = 1.0 / (math.sqrt(hb) * rho)
    M, n = O.act_multiplier(hb, 1.0, s_x)
    r = 1.0 / (math.sqrt(hb) * float(np.float32(s_x)))
    assert M * 127 * hb < 2 ** 30 and M < 2 ** 31 and M >= 2 ** 14
    assert abs(M - r * 2.0 ** n) <= 0.5
    M2 = int(np.rint(math.ldexp(r, n + 1)))
    assert M2 * 127 * hb >= 2 ** 30 or M2 >= 2 ** 31
    y = np.array([127 * hb, -127 * hb, 0, 1, -1])
    assert np.all(np.abs(M * y) + (1 << max(n - 1, 0)) < 2 ** 31)


def test_dynamic_multiplier_exact():
    for maxy in (1, 3, 127, 1000, 8191, 127 * 64):
        M, n = O.dynamic_multiplier(maxy, 64)
        assert abs(Fraction(M) - Fraction(127 * 2 ** n, maxy)) <= Fraction(1, 2)
        y = np.array([maxy, -maxy, 0])
        codes = np.clip(O.rshift_rne(M * y, n), -127, 127)
        assert list(codes) == [127, -127, 0]


# --------------------------------------------------------------- quantizers

def test_symmetric_quantizer():                                                # Eq. symmetric_q
    x = I.activations((1, 8, 8, 32), seed=41).astype(np.float64)
    s = O.symmetric_scale(x)
    q = O.quantize_sym(x, s)
    assert np.max(np.abs(q)) == 127 and q.min() >= -127
    assert np.max(np.abs(q * s - x)) <= s / 2 + 1e-12
    assert O.symmetric_scale(np.zeros(5)) == 1.0


def test_quantize_act_f16_is_quantized_transform():
    x = I.activations_f16((1, 4, 4, 128), seed=42)
    y = O.transform_real(x.astype(np.float64), 128)
    s = O.symmetric_scale(y)
    q = O.quantize_act_f16(x, 128, s).astype(np.int64)
    assert np.max(np.abs(q * s - y)) <= float(np.float32(s)) / 2 * (1 + 1e-6)


def test_quantize_act_i8_close_to_real_rescale():
    x = I.activations_i8((1, 6, 6, 192), seed=43, s_in=0.05)
    s_in = 0.05
    y = O.transform_real(x.astype(np.float64) * float(np.float32(s_in)), 64)
    s_x = float(np.float32(O.symmetric_scale(y)))
    q = O.quantize_act_i8(x, 64, s_in, s_x).astype(np.int64)
    exact = np.clip(np.rint(y / s_x), -127, 127)
    diff = np.abs(q - exact)
    assert diff.max() <= 1 and np.mean(diff > 0) < 1e-3


def test_quantize_act_dynamic():
    x = I.activations_i8((1, 5, 5, 64), seed=44, s_in=0.05)
    codes, s_used = O.quantize_act_dynamic_i8(x, 64, 0.05)
    assert np.max(np.abs(codes.astype(int))) == 127
    y = O.transform_real(x.astype(np.float64) * float(np.float32(0.05)), 64)
    assert math.isclose(s_used, np.max(np.abs(y)) / 127, rel_tol=1e-6)
    assert np.max(np.abs(codes * s_used - y)) <= s_used * 0.5001
    z, s0 = O.quantize_act_dynamic_i8(np.zeros((1, 2, 2, 64), np.int8), 64, 0.05)
    assert s0 == 1.0 and not z.any()
    xf = I.activations_f16((1, 3, 3, 128), seed=45)
    cf, sf = O.quantize_act_dynamic_f16(xf, 128)
    assert np.max(np.abs(cf.astype(int))) == 127
    assert math.isclose(sf, np.max(np.abs(O.transform_real(xf.astype(np.float64), 128))) / 127, rel_tol=1e-12)


# ---------------------------------------------------- integer transitions (golden table)

def test_transition_gammas_match_paper_table():
    tab = json.load(open(os.path.join(GOLDEN, "transitions.json")))["transitions"]
    m = 64
    val = {"1": 1.0, "sqrt(m)": math.sqrt(m)}
    w = I.weights(m, 1, 1, m, seed=50)
    for row in tab:
        form = row["from"]
        hb_next = m if row["to"] == "DH" else 0
        p = O.prepare_layer(w, None, form, m if form == "DH" else 0, m if form == "WH" else 0,
                            s_x=0.02, s_y=0.03, act="none", hb_next=hb_next, out_f32=False,
                            stride=1, pad=0)
        alpha = val[row["gamma_out"]] * val[row["gamma_in"]]
        expect = (float(np.float32(0.02)) * p.s_w) / (alpha * float(np.float32(0.03)))
        assert np.allclose(p.rho, expect, rtol=1e-15)
        assert (p.hb_out > 0) == (row["H_out"] == "H")
        assert (p.hb_next > 0) == (row["H_in"] == "H")


def _exact_transition(acc, p, rho_exact):
    """x_next = clamp(rint(H_in phi(H_out(rho (.) a)))) in exact rationals, from
    the real ratio rho (not M): the integer path may differ only through the
    M/2^n approximation of rho."""
    a = acc + p.b_int
    out = np.zeros(a.shape, dtype=np.int64)
    flat = a.reshape(-1, a.shape[-1])
    Hout = O.sylvester(p.hb_out) if p.hb_out else None
    Hin = O.sylvester(p.hb_next) if p.hb_next else None
    res = []
    for row in flat:
        t = [Fraction(float(r)) * int(v) for r, v in zip(rho_exact, row)]
        if Hout is not None:
            b = p.hb_out
            t = [sum(int(Hout[j % b][i]) * t[(j // b) * b + i] for i in range(b)) for j in range(len(t))]
        if p.act == "relu":
            t = [max(v, Fraction(0)) for v in t]
        if Hin is not None:
            b = p.hb_next
            t = [sum(int(Hin[j % b][i]) * t[(j // b) * b + i] for i in range(b)) for j in range(len(t))]
        res.append([max(-127, min(127, O.round_half_even_fraction(v))) for v in t])
    out[...] = np.array(res).reshape(a.shape)
    return out


@pytest.mark.parametrize("form,hb_next,act", [("DH", 0, "none"), ("DH", 16, "relu"), ("WH", 0, "relu"),
                                              ("WH", 16, "relu")])
def test_integer_transition_vs_exact_rational(form, hb_next, act):
    c = 32
    w = I.weights(c, 3, 3, 16, seed=60)
    b = I.bias(c, seed=61)
    x = I.activations_i8((1, 4, 4, 16), seed=62, s_in=0.05)
    def prep(s_y):
        return O.prepare_layer(w, b, form, 16 if form == "DH" else 0, 16 if form == "WH" else 0,
                               s_x=0.05, s_y=s_y, act=act, hb_next=hb_next, out_f32=False, stride=1, pad=1)
    p1 = prep(1.0)
    acc = O.conv_codes(x, p1.w_int, 1, 1)
    z = p1.rho * (acc + p1.b_int)                    # real-valued transition at s_y = 1
    z = O.transform_real(z, p1.hb_out, normalize=False) if p1.hb_out else z
    z = np.maximum(z, 0) if act == "relu" else z
    z = O.transform_real(z, hb_next, normalize=False) if hb_next else z
    p = prep(float(np.max(np.abs(z))) / 110.0)
    got = O.epilogue_int(acc, p).astype(np.int64)
    ref = _exact_transition(acc, p, p.rho)
    d = np.abs(got - ref)
    assert d.max() <= 1 and np.mean(d > 0) < 0.01
    assert np.mean(np.abs(ref) == 127) < 0.5                      # not saturated everywhere


@pytest.mark.parametrize("form", ["DH", "WH"])
def test_quantized_layer_approximates_real_layer(form):
    """End-to-end pin: dequantized integer output vs the fp64 real model."""
    c_in, c_out, hb = 64, 64, 64
    x_real = I.activations((1, 10, 10, c_in), seed=70).astype(np.float64)
    w = I.weights(c_out, 3, 3, c_in, seed=71)
    b = I.bias(c_out, seed=72)
    y_ref = np.maximum(O.conv_real(x_real, w, b, 1, 1), 0)
    s_x = O.symmetric_scale(O.transform_real(x_real, hb)) if form == "DH" else O.symmetric_scale(x_real)
    s_y = O.symmetric_scale(y_ref)
    p = O.prepare_layer(w, b, form, hb if form == "DH" else 0, hb if form == "WH" else 0, s_x, s_y,
                        "relu", 0, False, 1, 1)
    op = O.quantize_act_f16(x_real.astype(np.float16), hb if form == "DH" else 1, s_x)
    y = O.conv_layer(op, p).astype(np.float64) * p.s_y
    # WH keeps the outlier-heavy activations in the original domain (input
    # SQNR alone is ~24.5 dB here); DH quantizes them in the Hadamard domain.
    floor = 28.0 if form == "DH" else 20.0
    assert O.sqnr_db(y_ref, y) > floor
    pf = O.prepare_layer(w, b, form, hb if form == "DH" else 0, hb if form == "WH" else 0, s_x, s_y,
                         "relu", 0, True, 1, 1)
    yf = O.conv_layer(op, pf)
    assert O.sqnr_db(y_ref, yf) > floor


def test_chain_mixed_forms_tracks_real_model():
    """A small DH/WH chain with every transition of Table integer_transitions
    (WH-to-DH at 64 and 128 blocks, DH-to-WH) stays close to the real-valued
    model end to end."""
    from synth.configs import layer, ChainSpec
    layers = (layer("a", 16, 64, 3, 1, 1, "WH", "relu", hb_out=64),
              layer("b", 64, 64, 3, 2, 1, "DH", "relu", hb_in=64),
              layer("c", 64, 128, 3, 1, 1, "WH", "relu", hb_out=128),
              layer("d", 128, 32, 1, 1, 0, "DH", "none", hb_in=128))
    ch = ChainSpec("t", layers, 1, 12, 12, "i8", 0.05, 80, 81)
    assert O.transition_blocks(layers) == [64, 0, 128, 0]
    x = I.activations_i8((1, 12, 12, 16), seed=80, s_in=0.05)
    params = [(I.weights(L.c_out, L.k, L.k, L.c_in, 90 + i), I.bias(L.c_out, 95 + i)) for i, L in enumerate(layers)]
    x_real = x.astype(np.float64) * float(np.float32(0.05))
    scales = O.calibrate_chain(layers, params, x_real)
    preps = O.prepare_chain(layers, params, scales)
    outs = O.chain_forward(layers, preps, x, "i8", 0.05)
    ref = x_real
    for L, (w, b) in zip(layers, params):
        ref = O.conv_real(ref, w, b, L.stride, L.pad)
        ref = np.maximum(ref, 0) if L.act == "relu" else ref
    got = outs[-1].astype(np.float64) * preps[-1].s_y
    assert O.sqnr_db(ref, got) > 15.0


# ------------------------------------------------------- method diagnostics (T9)

def test_hadamard_domain_improves_tensorwise_sqnr_and_kurtosis():
    """Sec. transform-domain motivation: on outlier-heavy activations the
    Hadamard domain has lower excess kurtosis and higher per-tensor INT8 SQNR."""
    x = I.activations((1, 16, 16, 128), seed=0).astype(np.float64)
    y = O.transform_real(x, 128)
    qx = O.quantize_sym(x, O.symmetric_scale(x)) * O.symmetric_scale(x)
    qy = O.quantize_sym(y, O.symmetric_scale(y)) * O.symmetric_scale(y)
    assert O.sqnr_db(y, qy) > O.sqnr_db(x, qx)
    assert O.excess_kurtosis(y) < O.excess_kurtosis(x)


def test_range_expansion_indicator():
    """Eq. hadamard_sensitivity: a nonnegative, nonzero-mean tensor (ReLU
    output) expands under the transform; a zero-mean outlier tensor shrinks."""
    rng = np.random.default_rng(1)
    relu_like = np.maximum(rng.standard_normal((64, 64)) + 1.0, 0)
    assert O.range_expands(relu_like, 64)
    spiky = rng.standard_normal((64, 64)) * 0.1
    spiky[:, 3] = 50.0 * np.sign(rng.standard_normal(64))
    assert not O.range_expands(spiky, 64)


# ------------------------------------------------------- profiling (Eqs. hadamard_sensitivity, layerwise selection)

@pytest.mark.parametrize("hb", [2, 4, 16, 32, 64, 128])
def test_profile_constant_image_expands_by_sqrt_hb(hb):
    """Closed form: a constant code c (a nonzero channel mean) accumulates
    coherently into the constant basis, |T x|_inf = sqrt(hb) |c| > |c|."""
    x = np.full((1, 2, 3, 2 * hb), -5, np.int8)
    mx, mh, ind = O.range_expansion_codes(x, hb)
    assert mx[0] == 5 and mh[0] == 5 * hb and ind[0] == 1


@pytest.mark.parametrize("hb", [2, 8, 64, 256])
def test_profile_spike_shrinks_by_sqrt_hb(hb):
    """Closed form: one nonzero code per block spreads evenly, |T x|_inf =
    |c| / sqrt(hb) < |c|: no expansion."""
    x = np.zeros((1, 1, 2, hb), np.int8)
    x[0, 0, 0, 3 % hb] = 100
    x[0, 0, 1, 0] = -100
    mx, mh, ind = O.range_expansion_codes(x, hb)
    assert mx[0] == 100 and mh[0] == 100 and ind[0] == 0


def test_profile_ties_and_odd_orders_are_exact():
    """Strict '>' of Eq. hadamard_sensitivity on exact ties, and an odd power
    of two (sqrt(hb) irrational) decided without rounding."""
    tie = np.array([1, 1, 0, 0], np.int8).reshape(1, 1, 1, 4)      # T x = (1, 0, 1, 0): equal range
    assert O.range_expansion_codes(tie, 4)[2][0] == 0
    assert not O.range_expands(tie.astype(np.float64), 4)
    assert O.range_expansion_codes(np.array([1, 1], np.int8).reshape(1, 1, 1, 2), 2)[2][0] == 1   # sqrt2 > 1
    assert O.range_expansion_codes(np.array([3, -1], np.int8).reshape(1, 1, 1, 2), 2)[2][0] == 0  # 4/sqrt2 < 3
    assert O.range_expansion_codes(np.zeros((2, 1, 1, 16), np.int8), 16)[2].tolist() == [0, 0]


def test_profile_matches_dense_transform_per_image():
    """Brute force: the dense normalized transform in fp64 per image gives the
    same indicator wherever the two ranges are not within rounding of a tie."""
    rng = np.random.default_rng(7)
    x = rng.integers(-127, 128, size=(12, 3, 4, 64)).astype(np.int8)
    x[::3] = np.abs(x[::3])                      # nonnegative images: nonzero channel means
    x[1::3] = rng.integers(-2, 3, size=x[1::3].shape)              # small codes with one outlier channel:
    x[1::3, ..., 5] = 120                                          # the transform spreads the outlier
    mx, mh, ind = O.range_expansion_codes(x, 32)
    T = O.blockdiag_transform(64, 32)
    for k in range(x.shape[0]):
        xf = x[k].reshape(-1, 64).astype(np.float64)
        ref_h = np.abs(xf @ T.T).max()
        assert mx[k] == np.abs(xf).max()
        assert abs(mh[k] / math.sqrt(32) - ref_h) < 1e-9
        if abs(ref_h - mx[k]) > 1e-9:
            assert ind[k] == int(ref_h > mx[k])
    assert 0 < ind.sum() < len(ind)


def test_expansion_probability_and_selection():
    """p_l is the expanding fraction of the M images; pi_l = WH only when
    p_l > tau_sel (strict), with the paper's tau_sel = 0.8."""
    from fractions import Fraction
    assert O.expansion_probability([1, 1, 1, 1, 0]) == Fraction(4, 5)
    assert O.select_form(Fraction(4, 5)) == "DH"
    assert O.select_form(O.expansion_probability([1] * 5)) == "WH"
    assert O.select_form(Fraction(81, 100)) == "WH"
    assert O.select_form(Fraction(1, 2), tau=Fraction(1, 4)) == "WH"
    with pytest.raises(ValueError):
        O.expansion_probability([])


# ------------------------------------------------------- general nonlinearities (Sec. general nonlinearities)

@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_activation_lut_closed_forms(kind):
    """phi_int of Eq. supp_general_activation: phi(0) = 0, the printed values
    SiLU(1) = 0.7310585786300049 and GELU(1) = 0.8413447460685429, and the
    identity phi(v) - phi(-v) = v shared by SiLU and GELU (two roundings:
    within one code wherever the table does not clamp)."""
    s_z, s_u = 1.0 / 64, 1.0 / 100
    lut = O.activation_lut(kind, s_z, s_u)
    assert lut[127] == 0
    assert lut[127 + 64] == {"silu": 73, "gelu": 84}[kind]
    for z in range(1, 128):
        up, dn = int(lut[127 + z]), int(lut[127 - z])
        if abs(up) < 127 and abs(dn) < 127:
            assert abs((up - dn) - s_z * z / s_u) <= 1.0
    assert all(lut[127 + z] <= lut[127 + z + 1] for z in range(0, 126))   # increasing for v >= 0


def _general_case(form, hb_next, kind, seed=0):
    c_in, c_out = 64, 64
    x_real = np.maximum(I.activations((1, 8, 9, c_in), seed=seed + 80).astype(np.float64), 0)
    w = I.weights(c_out, 3, 3, c_in, seed=seed + 81)
    b = I.bias(c_out, seed=seed + 82)
    hb_in, hb_out = (64, 0) if form == "DH" else (0, 64)
    y_lin = O.conv_real(x_real, w, b, 1, 1)
    phi = np.vectorize(lambda v: O.phi(kind, v))
    u_real = phi(y_lin)
    s_x = O.symmetric_scale(O.transform_real(x_real, 64)) if form == "DH" else O.symmetric_scale(x_real)
    s_z = O.symmetric_scale(y_lin)
    s_u = O.symmetric_scale(u_real)
    target = O.transform_real(u_real, hb_next) if hb_next else u_real
    s_y = O.symmetric_scale(target)
    p = O.prepare_layer(w, b, form, hb_in, hb_out, s_x, s_y, kind, hb_next, False, 1, 1, s_z=s_z, s_u=s_u)
    op = O.quantize_act_f16(x_real.astype(np.float16), hb_in if form == "DH" else 1, s_x)
    return p, op, target, y_lin


@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_general_transition_matches_its_equations_step_by_step(kind):
    """With s_u = s_y and no next transform the input-side rescale is exactly
    2^n_in / 2^n_in, so the output codes are phi_int(z); z is recomputed here
    from exact rationals of H~_out (M_out (.) a) / 2^n_out and phi_int from
    the activation formula itself (not the table)."""
    p, op, _, _ = _general_case("WH", 0, kind)
    p.M_in, p.n_in = O.fixed_point([1.0], [127], 1)
    p.M_in = int(p.M_in[0])
    assert p.M_in == 2 ** p.n_in
    got = O.conv_layer(op, p).astype(np.int64)
    acc = O.conv_codes(op, p.w_int, 1, 1) + p.b_int
    H = O.sylvester(64)
    for (i, j) in [(0, 0), (3, 5), (7, 8)]:
        a = [int(v) for v in acc[0, i, j]]
        t = [int(m) * v for m, v in zip(p.M, a)]
        for c in (0, 17, 63):
            v = sum(int(H[c, k]) * t[k] for k in range(64))
            z = min(max(O.round_half_even_fraction(Fraction(v, 2 ** p.n)), -127), 127)
            u = min(max(int(round(O.phi(kind, p.s_z * z) / p.s_u)), -127), 127)
            assert got[0, i, j, c] == u


@pytest.mark.parametrize("form,hb_next,kind", [("DH", 0, "silu"), ("WH", 0, "gelu"), ("DH", 64, "gelu"),
                                               ("WH", 32, "silu")])
def test_general_transition_tracks_real_model(form, hb_next, kind):
    """End to end: the two-step integer transition (preactivation codes, table,
    fixed-point rescale with the fused next transform) stays close to the
    fp64 model phi(conv) (and its next-layer transform)."""
    p, op, target, _ = _general_case(form, hb_next, kind, seed=3)
    y = O.conv_layer(op, p).astype(np.float64) * p.s_y
    assert O.sqnr_db(target, y) > (24.0 if form == "DH" else 18.0)
    assert np.mean(np.abs(O.conv_layer(op, p)) == 127) < 0.1


# ------------------------------------------------------- paper-exact orders (Supp. Hadamard construction)

def test_every_supported_order_is_a_hadamard_matrix():
    """Eq. hadamard_properties for every order of M_H up to 256: entries +-1
    and H~ H~^T = m I (Sylvester, Paley-I, Paley-II, Kronecker products)."""
    orders = O.supported_orders(256)
    assert {4, 8, 12, 20, 24, 28, 36, 44, 192, 224, 240} <= set(orders)
    for m in orders:
        H = O.hadamard_of_order(m, orders)
        assert H.shape == (m, m) and np.all(np.abs(H) == 1)
        assert np.array_equal(H @ H.T, m * np.eye(m, dtype=np.int64)), m


def test_paley_constructions_closed_forms():
    """Paley-I (q = 3 mod 4) gives order q + 1 from an antisymmetric Jacobsthal
    matrix, Paley-II (q = 1 mod 4) order 2 (q + 1) from a symmetric one; both
    reject the other residue class."""
    Q7 = O._jacobsthal(7)
    assert np.array_equal(Q7, -Q7.T) and np.all(Q7.sum(axis=1) == 0)
    Q13 = O._jacobsthal(13)
    assert np.array_equal(Q13, Q13.T)
    assert O.paley1(7).shape == (8, 8) and O.paley2(13).shape == (28, 28)
    for bad in (lambda: O.paley1(13), lambda: O.paley2(7), lambda: O.paley1(15)):
        with pytest.raises(ValueError):
            bad()


def test_hadamard_order_rule():
    """Eq. hadamard_order: m(C) = min supported order >= 4 ceil(C / 4); the
    orders the paper names: m(192) = 192 (Paley-I, q = 191), m(224) = 224
    (q = 223), m(320) = 320 (a Kronecker product)."""
    assert O.hadamard_order(192) == 192 and O.supported_orders(256)[192] == ("paley1", 191)
    assert O.hadamard_order(224) == 224 and O.supported_orders(256)[224] == ("paley1", 223)
    assert O.hadamard_order(320) == 320 and O.supported_orders(512)[320][0] == "kron"
    assert O.hadamard_order(3) == 4 and O.hadamard_order(13) == 16 and O.hadamard_order(100) == 104
    for c in range(1, 300, 7):
        m = O.hadamard_order(c)
        assert m >= 4 * ((c + 3) // 4)
        assert not any(4 * ((c + 3) // 4) <= k < m for k in O.supported_orders(512))


@pytest.mark.parametrize("c", [3, 20, 100, 192, 200])
def test_padded_transforms_are_semi_orthogonal_and_preserve_the_layer(c):
    """Eqs. supp_padded_transforms, supp_semi_orthogonality: T T^T = I_C for
    both orientations, so DH (X T_in)(W T_in)^T and WH (X (T_out^T W)^T) T_out^T
    both reproduce X W^T with padding to m(C)."""
    T_in, T_out = O.padded_transforms(c)
    m = O.hadamard_order(c)
    assert T_in.shape == (c, m) and T_out.shape == (c, m)
    assert np.allclose(T_in @ T_in.T, np.eye(c), atol=1e-12)
    assert np.allclose(T_out @ T_out.T, np.eye(c), atol=1e-12)
    rng = np.random.default_rng(c)
    X = rng.standard_normal((5, c))
    W = rng.standard_normal((7, c))
    assert np.allclose((X @ T_in) @ (W @ T_in).T, X @ W.T, atol=1e-10)
    Wo = rng.standard_normal((c, 6))                         # C_out = c rows
    Xo = rng.standard_normal((4, 6))
    Wbar = T_out.T @ Wo                                      # m x C_in
    assert np.allclose((Xo @ Wbar.T) @ T_out.T, Xo @ Wo.T, atol=1e-10)


def test_construction_rule_prefers_paley1_and_smallest_kronecker_factor():
    """Reading R9: Paley-I before Paley-II where both exist (12 = Paley-I(11),
    not Paley-II(5)); Paley-II where Paley-I does not (28, q = 13); a product
    order takes the smallest supported left factor (320 = H~_2 (x) H~_160)."""
    o = O.supported_orders(1024)
    assert o[12] == ("paley1", 11) and o[28] == ("paley2", 13) and o[36] == ("paley2", 17)
    assert o[320] == ("kron", 2, 160) and o[160] == ("kron", 2, 80) and o[80] == ("paley1", 79)
    assert np.array_equal(O.hadamard_of_order(320), np.kron(O.sylvester(4), O.paley1(79)))


def test_paley1_transform_of_a_constant_vector():
    """Closed form that fixes the orientation: with H~ = I + S, S = [[0, 1^T],
    [-1, Q]] and zero column sums of the Jacobsthal matrix Q, the input-side
    transform y_j = sum_i H~[i][j] x_i of x = mu 1 is mu (2 - m) at j = 0 and
    2 mu elsewhere (the transposed matrix would give mu m, 0, ..., 0)."""
    m, mu = 192, 3
    y = O.transform_order_int(np.full((2, m), mu, np.int8), m)
    assert np.all(y[:, 0] == mu * (2 - m)) and np.all(y[:, 1:] == 2 * mu)
    yr = O.transform_order_real(np.full((1, m), 1.0), m) * math.sqrt(m)
    assert np.allclose(yr[0, 0], 2 - m) and np.allclose(yr[0, 1:], 2.0)


@pytest.mark.parametrize("c", [20, 100, 190, 192, 320])
def test_order_transforms_are_semi_orthogonal_and_exact(c):
    """Eq. supp_semi_orthogonality for the loop-order transform
    (rows of T_in = P_C H_m orthonormal), the padded DH identity of
    Eq. supp_padded_dh, and the integer transform equal to sqrt(m) times the
    real one on codes."""
    m = O.hadamard_order(c)
    T = O.transform_order_real(np.eye(c), m)
    assert T.shape == (c, m) and np.allclose(T @ T.T, np.eye(c), atol=1e-12)
    rng = np.random.default_rng(c)
    x = rng.standard_normal((1, 6, 5, c))
    w = rng.standard_normal((4, 3, 3, c))
    assert np.allclose(O.conv_real(O.transform_order_real(x, m), O.transform_order_real(w, m), None, 1, 1),
                       O.conv_real(x, w, None, 1, 1), atol=1e-10)
    codes = rng.integers(-127, 128, size=(3, 7, c)).astype(np.int8)
    yi = O.transform_order_int(codes, m)
    assert np.array_equal(yi.astype(np.float64), np.rint(O.transform_order_real(codes, m) * math.sqrt(m)))


def test_order_quantizer_tracks_the_real_quantizer():
    """INT8 entry into the order-m basis: equal to the real-valued quantizer
    Q(x T_in) up to the (M, n) approximation (at most one code, rarely), zero
    stays zero, and the codes span the range."""
    c, m, s_in = 190, 192, 0.05
    x = I.activations_i8((2, 9, 11, c), seed=41, s_in=s_in)
    y_real = O.transform_order_real(x.astype(np.float64) * float(np.float32(s_in)), m)
    s_x = float(np.float32(O.symmetric_scale(y_real)))
    got = O.quantize_act_order_i8(x, m, s_in, s_x).astype(np.int64)
    ref = O.quantize_sym(y_real, s_x)
    d = np.abs(got - ref)
    assert got.shape[-1] == m and d.max() <= 1 and np.mean(d > 0) < 1e-3
    assert np.abs(got).max() == 127
    assert not O.quantize_act_order_i8(np.zeros((1, 2, 2, c), np.int8), m, s_in, s_x).any()


def test_order_layer_tracks_the_real_model():
    """A DH layer in the paper's order (Eq. supp_padded_dh) on the quantized
    operand stays close to the fp64 model."""
    c = 190
    m = O.hadamard_order(c)
    x_real = np.maximum(I.activations((1, 12, 12, c), seed=42).astype(np.float64), 0)
    w, b = I.weights(64, 3, 3, c, seed=43), I.bias(64, seed=44)
    y_ref = O.conv_real(x_real, w, b, 1, 1)
    s_in = float(np.float32(O.symmetric_scale(x_real)))
    x_i8 = O.quantize_sym(x_real, s_in).astype(np.int8)
    s_x = float(np.float32(O.symmetric_scale(O.transform_order_real(x_real, m))))
    p = O.prepare_layer(w, b, "DH", 0, 0, s_x, float(np.float32(O.symmetric_scale(y_ref))), "none", 0, False, 1, 1,
                        order_in=m)
    assert p.w_int.shape == (64, 3, 3, m)
    y = O.conv_layer(O.quantize_act_order_i8(x_i8, m, s_in, s_x), p).astype(np.float64) * p.s_y
    # against the model on the INT8 input it was given (transform-domain and weight quantization only),
    # and against the model on the real input (plus the original-domain input quantization)
    assert O.sqnr_db(O.conv_real(x_i8.astype(np.float64) * s_in, w, b, 1, 1), y) > 25.0
    assert O.sqnr_db(y_ref, y) > 18.0


# ------------------------------------------------------- decoder-side operators (transposed, sub-pixel)

@pytest.mark.parametrize("k,stride,pad", [(5, 2, 2), (3, 2, 1), (3, 1, 1), (1, 1, 0)])
def test_transposed_conv_is_the_adjoint_of_the_strided_conv(k, stride, pad):
    """<F x, z> = <x, F^T z>: the transposed convolution with the channel-
    transposed weights is the adjoint of the forward convolution."""
    rng = np.random.default_rng(k * 10 + stride)
    x = rng.standard_normal((2, 7, 9, 5))
    w = rng.standard_normal((6, k, k, 5))
    y = O.conv_real(x, w, None, stride, pad)
    z = rng.standard_normal(y.shape)
    ho, wo = O.conv_transpose_hw(y.shape[1], y.shape[2], k, stride, pad)
    xt = O.conv_transpose_real(z, w.transpose(3, 1, 2, 0), None, stride, pad,
                               out_pad=max(0, 7 - ho))[:, :7, :9, :]
    assert xt.shape == x.shape
    assert abs(np.sum(y * z) - np.sum(x * xt)) < 1e-9 * max(1.0, abs(np.sum(y * z)))


def test_transposed_conv_stride1_is_a_flipped_forward_conv_and_codes_are_exact():
    """Closed form: stride 1 and padding p equal a forward convolution with the
    spatially flipped kernel and padding k - 1 - p; on integer codes the int64
    scatter equals the fp64 one exactly."""
    rng = np.random.default_rng(3)
    x = rng.integers(-127, 128, size=(1, 6, 8, 4))
    w = rng.integers(-127, 128, size=(5, 3, 3, 4))
    ref = O.conv_real(x, w[:, ::-1, ::-1, :], None, 1, 1)
    got = O.conv_transpose_real(x, w, None, 1, 1)
    assert np.array_equal(got, ref)
    assert np.array_equal(O.conv_transpose_codes(x, w, 2, 1, 1), O.conv_transpose_real(x, w, None, 2, 1, 1))


@pytest.mark.parametrize("form", ["DH", "WH"])
def test_transposed_conv_preserves_function_in_both_forms(form):
    """Eq. linear_operator holds for the transposed operator too: DH transforms
    the contracted C_in of activations and weights, WH the weights' C_out with
    the output basis restored afterwards; both reproduce the layer."""
    rng = np.random.default_rng(5)
    x = rng.standard_normal((1, 5, 6, 64))
    w = rng.standard_normal((32, 5, 5, 64)) * 0.1
    b = rng.standard_normal(32) * 0.1
    ref = O.conv_transpose_real(x, w, b, 2, 2, 1)
    if form == "DH":
        wp, bb = O.transform_weights(w, b, "DH", 64, 0)
        got = O.conv_transpose_real(O.transform_real(x, 64), wp, bb, 2, 2, 1)
    else:
        wp, bb = O.transform_weights(w, b, "WH", 0, 32)
        got = O.transform_real(O.conv_transpose_real(x, wp, bb, 2, 2, 1), 32)
    assert np.allclose(got, ref, atol=1e-10)


def test_quantized_transposed_layer_tracks_real_model():
    """A DH synthesis layer (5x5, stride 2, 64 -> 32) on INT8 codes with the
    integer transition stays close to the fp64 transposed convolution."""
    x_real = I.activations((1, 8, 9, 64), seed=90).astype(np.float64)
    w = I.weights(32, 5, 5, 64, seed=91)
    b = I.bias(32, seed=92)
    y_ref = np.maximum(O.conv_transpose_real(x_real, w, b, 2, 2, 1), 0)
    s_x = O.symmetric_scale(O.transform_real(x_real, 64))
    s_y = O.symmetric_scale(y_ref)
    p = O.prepare_layer(w, b, "DH", 64, 0, s_x, s_y, "relu", 0, False, 2, 2)
    op = O.quantize_act_f16(x_real.astype(np.float16), 64, s_x)
    y = O.conv_transpose_layer(op, p, 1).astype(np.float64) * p.s_y
    assert y.shape == y_ref.shape
    assert O.sqnr_db(y_ref, y) > 28.0


def test_depth_to_space_index_mapping():
    """Sub-pixel rearrangement: channel c r^2 + i r + j goes to pixel
    (h r + i, w r + j), channel c; space_to_depth inverts it."""
    x = np.arange(8).reshape(1, 1, 1, 8)                 # c = 2, r = 2
    y = O.depth_to_space(x, 2)
    assert y.shape == (1, 2, 2, 2)
    assert y[0, :, :, 0].tolist() == [[0, 1], [2, 3]] and y[0, :, :, 1].tolist() == [[4, 5], [6, 7]]
    z = np.random.default_rng(0).integers(0, 9, size=(2, 3, 4, 18))
    assert np.array_equal(O.space_to_depth(O.depth_to_space(z, 3), 3), z)


# ------------------------------------------------------- dynamic affine activation quantization (PTQ)

def test_affine_params_closed_forms():
    """Eq. affine_q: s = (max' - min') / 255 and z = round(-min' / s), zero
    representable exactly; a nonnegative tensor gets z = 0; a zero tensor
    (1, 0); dequantization error at most s / 2 in range (Eq. uniform_q)."""
    x = np.array([-1.0, 0.0, 0.5, 2.0])
    s, z = O.affine_params(x)
    assert s == pytest.approx(3.0 / 255) and z == 85
    q = O.quantize_affine(x, s, z)
    assert q[1] == z and s * (q[1] - z) == 0.0
    assert np.all(np.abs(s * (q - z) - x) <= s / 2 + 1e-12)
    assert O.affine_params(np.array([0.2, 3.0])) == pytest.approx((3.0 / 255, 0))
    assert O.affine_params(np.array([-4.0, -1.0]))[1] == 255
    assert O.affine_params(np.zeros(5)) == (1.0, 0)


def test_wide_code_conv_matches_the_int8_conv_and_fp64():
    """conv_codes_wide equals the nested-loop C convolution on INT8 codes and
    the fp64 convolution on centred codes up to +-255 (exact integers)."""
    rng = np.random.default_rng(4)
    x8 = rng.integers(-127, 128, size=(2, 7, 6, 16)).astype(np.int8)
    w = rng.integers(-127, 128, size=(8, 3, 3, 16)).astype(np.int8)
    assert np.array_equal(O.conv_codes_wide(x8, w, 2, 1), O.conv_codes(x8, w, 2, 1))
    xw = rng.integers(-255, 256, size=(1, 5, 5, 16))
    assert np.array_equal(O.conv_codes_wide(xw, w, 1, 1), O.conv_real(xw, w, None, 1, 1).astype(np.int64))


@pytest.mark.parametrize("form", ["DH", "WH"])
def test_dynamic_affine_layer_tracks_real_model_and_pads_with_centred_zero(form):
    """The PTQ layer: dynamic (s, z) per input, MACs on centred codes,
    dequantized output; it tracks the fp64 model, and a zero-padded border
    sees the centred zero (the result equals the layer on an explicitly
    zero-padded input without padding)."""
    x_real = I.activations((1, 9, 10, 64), seed=120).astype(np.float64) + 1.5     # shifted, nonzero mean
    w = I.weights(32, 3, 3, 64, seed=121)
    b = I.bias(32, seed=122)
    hb_in, hb_out = (64, 0) if form == "DH" else (0, 32)
    p = O.prepare_layer(w, b, form, hb_in, hb_out, 1.0, 1.0, "none", 0, True, 1, 1)
    y, s, z = O.conv_layer_affine(x_real, p)
    y_ref = O.conv_real(x_real, w, b, 1, 1)
    assert O.sqnr_db(y_ref, y) > (30.0 if form == "DH" else 22.0)
    assert z != 0 or form == "WH"
    xp = np.zeros((1, 11, 12, 64))
    xp[:, 1:10, 1:11, :] = x_real
    p0 = O.prepare_layer(w, b, form, hb_in, hb_out, 1.0, 1.0, "none", 0, True, 1, 0)
    y0, s0, z0 = O.conv_layer_affine(xp, p0)
    assert (s0, z0) == (s, z) or form == "WH"
    if form == "DH":
        assert np.allclose(y0, y, atol=1e-9)


# ------------------------------------------------------- GDN / IGDN (channel-coupled nonlinearities)

def test_gdn_closed_forms():
    """gamma = 0: v / sqrt(beta); diagonal gamma: elementwise v / sqrt(beta +
    g v^2); IGDN inverts GDN when the normalization does not depend on v
    (gamma = 0), and a single channel satisfies IGDN(GDN(v)) = v exactly in
    closed form v / r * sqrt(beta + g (v / r)^2) with r = sqrt(beta + g v^2)."""
    v = np.array([[0.5, -2.0, 3.0]])
    beta = np.array([1.0, 4.0, 0.25])
    assert np.allclose(O.gdn(v, beta, np.zeros((3, 3))), v / np.sqrt(beta))
    g = np.diag([0.5, 1.0, 2.0])
    assert np.allclose(O.gdn(v, beta, g), v / np.sqrt(beta + np.diag(g) * v * v))
    assert np.allclose(O.gdn(O.gdn(v, beta, np.zeros((3, 3))), beta, np.zeros((3, 3)), inverse=True), v)
    one = O.gdn(np.array([[2.0]]), [1.0], [[0.75]])
    assert one[0, 0] == pytest.approx(2.0 / math.sqrt(1.0 + 0.75 * 4.0))
    assert np.allclose(O.gdn(v, beta, g, inverse=True), v * np.sqrt(beta + np.diag(g) * v * v))


@pytest.mark.parametrize("inverse", [False, True])
def test_gdn_transition_tracks_real_model(inverse):
    """A DH layer followed by GDN (or IGDN) through the two-step integer
    transition stays close to the fp64 model gdn(conv(x))."""
    rng = np.random.default_rng(9)
    c = 64
    x_real = np.maximum(I.activations((1, 7, 8, c), seed=130).astype(np.float64), 0)
    w = I.weights(c, 3, 3, c, seed=131)
    b = I.bias(c, seed=132)
    beta = 1.0 + rng.random(c)
    gamma = np.abs(rng.standard_normal((c, c))) * 0.01
    y = O.conv_real(x_real, w, b, 1, 1)
    u = O.gdn(y, beta, gamma, inverse)
    s_x = O.symmetric_scale(O.transform_real(x_real, 64))
    s_z, s_u = O.symmetric_scale(y), O.symmetric_scale(u)
    p = O.prepare_layer(w, b, "DH", 64, 0, s_x, s_u, "igdn" if inverse else "gdn", 0, False, 1, 1,
                        s_z=s_z, s_u=s_u, gdn_beta=beta, gdn_gamma=gamma)
    op = O.quantize_act_f16(x_real.astype(np.float16), 64, s_x)
    acc = O.conv_codes(op, p.w_int, 1, 1)
    got = O.epilogue_general_vector(acc, p).astype(np.float64) * p.s_y
    assert O.sqnr_db(u, got) > 24.0


def _round_half_away(x):
    return np.sign(x) * np.floor(np.abs(x) + 0.5)


def _gdn_case(c, seed, inverse, gamma_scale=0.01):
    rng = np.random.default_rng(seed)
    beta = 0.5 + rng.random(c)
    gamma = np.abs(rng.standard_normal((c, c))) * gamma_scale
    z = rng.integers(-127, 128, (400, c))
    z[0] = 127
    z[1] = 0
    z[2, : c // 2] = -127
    s_z = 0.04
    y = O.gdn(s_z * z.astype(np.float64), beta, gamma, inverse)
    s_u = float(np.float32(np.abs(y).max() / 120.0))
    return beta, gamma, z, s_z, s_u, y


@pytest.mark.parametrize("inverse", [False, True])
@pytest.mark.parametrize("c", [16, 64, 192])
def test_gdn_int_rounds_the_real_gdn(inverse, c):
    """R21: phi_int(z) is round(phi(s_z z) / s_u) up to the 9-bit pool
    coefficients and the fixed-point R^2: never more than one code away from
    the fp64 model, equal on at least 97% of the codes, and the pool
    parameters respect their bounds."""
    beta, gamma, z, s_z, s_u, y = _gdn_case(c, 40 + c, inverse)
    g = O.gdn_params(beta, gamma, s_z, s_u, inverse)
    assert g.G.max() <= 511 and g.d_max < 2 ** 31 and g.P >= 2 ** 15
    assert g.G.max() >= 256                                     # e is the largest admissible
    u = O.gdn_int(z, g)
    ref = np.clip(_round_half_away(y / s_u), -127, 127)
    d = np.abs(u - ref)
    assert d.max() <= 1 and np.mean(d > 0) < 0.03
    assert np.abs(u).max() >= 118


def test_gdn_int_is_the_largest_admissible_code():
    """Brute force on three channels: |u| is the largest k in [0, 127] with
    (2k - 1)^2 D 2^t <= 4 P z^2 (GDN) / (2k - 1)^2 2^t <= 4 P z^2 D (IGDN),
    found by trying every k with Python integers; D itself by the definition
    B_i + sum_j G_ij z_j^2 written out term by term."""
    rng = np.random.default_rng(3)
    beta = np.array([0.7, 1.3, 0.2])
    gamma = np.array([[0.1, 0.02, 0.0], [0.03, 0.2, 0.05], [0.0, 0.01, 0.3]])
    for inverse in (False, True):
        g = O.gdn_params(beta, gamma, 0.05, 0.012 if not inverse else 0.05, inverse)
        z = rng.integers(-127, 128, (60, 3))
        u = O.gdn_int(z, g)
        for r in range(z.shape[0]):
            for i in range(3):
                D = int(g.B[i]) + sum(int(g.G[i, j]) * int(z[r, j]) ** 2 for j in range(3))
                zi = int(z[r, i])
                best = 0
                for k in range(1, 128):
                    lhs = (2 * k - 1) ** 2 * (2 ** g.t if inverse else D * 2 ** g.t)
                    rhs = 4 * g.P * zi * zi * (D if inverse else 1)
                    if lhs <= rhs:
                        best = k
                assert int(u[r, i]) == (best if zi >= 0 else -best)


def test_gdn_int_gamma_zero_and_symmetries():
    """gamma = 0: the pool is beta alone, u = round(s_z z / (s_u sqrt(beta)))
    within one code; phi_int is odd in z; permuting the channels of z, beta
    and gamma permutes u; IGDN of the GDN codes returns z within 2 codes
    when gamma = 0 (the two roots cancel)."""
    c = 8
    beta = np.linspace(0.5, 2.0, c)
    z = np.random.default_rng(5).integers(-127, 128, (200, c))
    g0 = O.gdn_params(beta, np.zeros((c, c)), 0.05, 0.05 / np.sqrt(0.5), False)
    u = O.gdn_int(z, g0)
    ref = _round_half_away(0.05 * z / (0.05 / np.sqrt(0.5) * np.sqrt(beta)))
    assert np.abs(u - np.clip(ref, -127, 127)).max() <= 1
    assert np.array_equal(O.gdn_int(-z, g0), -u)
    inv = O.gdn_params(beta, np.zeros((c, c)), 0.05 / np.sqrt(0.5), 0.05, True)
    assert np.abs(O.gdn_int(u, inv) - z).max() <= 2
    beta2, gamma2, z2, s_z, s_u, _ = _gdn_case(c, 7, False, 0.05)
    g = O.gdn_params(beta2, gamma2, s_z, s_u)
    perm = np.random.default_rng(8).permutation(c)
    gp = O.gdn_params(beta2[perm], gamma2[np.ix_(perm, perm)], s_z, s_u)
    assert np.array_equal(O.gdn_int(z2[:, perm], gp), O.gdn_int(z2, g)[:, perm])


def test_gdn_params_reject_invalid():
    with pytest.raises(ValueError):
        O.gdn_params([1.0, 0.0], np.zeros((2, 2)), 0.1, 0.1)
    with pytest.raises(ValueError):
        O.gdn_params([1.0, 1.0], -np.ones((2, 2)), 0.1, 0.1)
    with pytest.raises(ValueError):
        O.gdn_params([1.0, 1.0], np.zeros((3, 3)), 0.1, 0.1)
