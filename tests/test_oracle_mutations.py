"""Plants plausible mistakes in the CPU oracle (on the CPU, via monkeypatch)
and checks that at least one pin in test_oracle_pins.py catches each of
them: a dropped term, a wrong sign or index, a transposed operand, a wrong
normalization or rounding."""
import math

import numpy as np
import pytest

import tests.test_oracle_pins as P
from oracle import hatq_oracle as O

_orig = {k: getattr(O, k) for k in ("sylvester", "transform_real", "transform_int", "rshift_rne",
                                    "fixed_point", "prepare_layer", "epilogue_int", "conv_codes",
                                    "quantize_act_i8", "transform_weights", "quantize_sym",
                                    "act_multiplier", "range_expansion_codes", "select_form",
                                    "epilogue_general", "phi", "paley1", "padded_transforms",
                                    "_jacobsthal", "conv_transpose_codes", "conv_transpose_real",
                                    "depth_to_space", "affine_params", "conv_layer_affine", "gdn", "gdn_pool", "gdn_int",
                                    "transform_order_real", "transform_order_int", "quantize_act_order_i8",
                                    "hadamard_of_order")}


def _sylvester_bad(m):
    H = _orig["sylvester"](m).copy()
    if m >= 4:
        H[-1, 1] *= -1
    return H


def _transform_real_bad(x, hb, normalize=True):
    y = _orig["transform_real"](x, hb, normalize=False)
    return y / hb if normalize and hb > 1 else y


def _transform_int_bad(x, hb):
    y = _orig["transform_int"](x, hb)
    if hb > 1:
        y = y.reshape(-1, y.shape[-1])
        y[:, 1] = -y[:, 1]
    return y.reshape(np.shape(x))


def _rshift_floor(v, n):
    return np.asarray(v, dtype=np.int64) >> n


def _fixed_point_no_gain(rho, a_bound, gain=1):
    return _orig["fixed_point"](rho, a_bound, 1)


def _prepare_no_gamma_in(*a, **k):
    p = _orig["prepare_layer"](*a, **k)
    if getattr(p, "rho", None) is not None and p.hb_next:
        p.rho = p.rho * math.sqrt(p.hb_next)
    return p


def _epilogue_m_after_h(acc, p):
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    v = O.transform_int(a, p.hb_out) if p.hb_out else a
    t = p.M * v
    u = np.maximum(t, 0) if p.act == "relu" else t
    w = O.transform_int(u, p.hb_next) if p.hb_next else u
    return np.clip(O.rshift_rne(w, p.n), -127, 127).astype(np.int8)


def _epilogue_no_bias(acc, p):
    class Q:
        pass
    q = Q()
    q.__dict__.update(p.__dict__)
    q.b_int = np.zeros_like(p.b_int)
    return _orig["epilogue_int"](acc, q)


def _conv_swap(x, w, stride, pad, window=None):
    return _orig["conv_codes"](x, w, pad if pad else stride, stride, window)


def _act_mult_no_sqrt(hb, s_in, s_x):
    rho = float(np.float32(s_in)) / float(np.float32(s_x))
    M, n = O.fixed_point([rho], [127 * hb], 1)
    return int(M[0]), n


def _wh_wrong_axis(w_ohwi, b, form, hb_in, hb_out):
    if form == "WH":
        w = np.asarray(w_ohwi, dtype=np.float64)
        hb = min(hb_out, w.shape[-1] & -w.shape[-1])
        return O.transform_real(w, hb), O.transform_real(np.asarray(b, np.float64), hb_out)
    return _orig["transform_weights"](w_ohwi, b, form, hb_in, hb_out)


def _quantize_floor(x, s):
    return np.clip(np.floor(np.asarray(x, dtype=np.float64) / s), -127, 127).astype(np.int64)


def _profile_non_strict(x_i8, hb):
    mx, mh, _ = _orig["range_expansion_codes"](x_i8, hb)
    return mx, mh, np.array([int(h) ** 2 >= hb * int(m) ** 2 for h, m in zip(mh, mx)], np.uint8)


def _profile_unnormalized(x_i8, hb):
    mx, mh, _ = _orig["range_expansion_codes"](x_i8, hb)
    return mx, mh, np.array([int(h) > int(m) for h, m in zip(mh, mx)], np.uint8)


def _select_non_strict(p, tau=None):
    from fractions import Fraction
    tau = Fraction(4, 5) if tau is None else Fraction(tau)
    return "WH" if Fraction(p) >= tau else "DH"


def _general_h_before_m(acc, p):
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    v = O.transform_int(a, p.hb_out) if p.hb_out else a
    t = p.M * v
    z = np.clip(O.rshift_rne(t, p.n), -127, 127)
    w = p.M_in * p.lut[z + 127]
    w = O.transform_int(w, p.hb_next) if p.hb_next else w
    return np.clip(O.rshift_rne(w, p.n_in), -127, 127).astype(np.int8)


def _general_lut_shifted(acc, p):
    q = O.Prepared(**p.__dict__)
    q.lut = np.concatenate([p.lut[1:], p.lut[-1:]])
    return _orig["epilogue_general"](acc, q)


def _phi_sign(kind, v):
    return v / (1.0 + math.exp(v)) if kind == "silu" else _orig["phi"](kind, -v)


def _paley1_no_identity(q):
    return _orig["paley1"](q) - np.eye(q + 1, dtype=np.int64)


def _jacobsthal_chi0(q):
    Q = _orig["_jacobsthal"](q).copy()
    np.fill_diagonal(Q, 1)
    return Q


def _padded_unnormalized(c):
    T_in, T_out = _orig["padded_transforms"](c)
    m = T_in.shape[1]
    return T_in * math.sqrt(m), T_out * math.sqrt(m)


def _convT_gather(x, w, stride, pad, out_pad=0):
    # a forward-style gather with the transposed output size (the classic mix-up)
    y = O.conv_codes(x, w, 1, pad)
    ho, wo = O.conv_transpose_hw(x.shape[1], x.shape[2], w.shape[1], stride, pad, out_pad)
    out = np.zeros((x.shape[0], ho, wo, w.shape[0]), np.int64)
    hh, ww = min(ho, y.shape[1]), min(wo, y.shape[2])
    out[:, :hh, :ww] = y[:, :hh, :ww]
    return out


def _convT_real_unflipped_pad(x, w, b, stride, pad, out_pad=0):
    return _orig["conv_transpose_real"](x, w, b, stride, max(pad - 1, 0), out_pad)[:, :, :, :] if pad else \
        _orig["conv_transpose_real"](x, w, b, stride, pad, out_pad) * 1.0001


def _d2s_swapped(x, r):
    x = np.asarray(x)
    n, h, w, crr = x.shape
    c = crr // (r * r)
    return x.reshape(n, h, w, r, r, c).transpose(0, 1, 3, 2, 4, 5).reshape(n, h * r, w * r, c)


def _affine_z_sign(x):
    s, z = _orig["affine_params"](x)
    lo = min(float(np.min(x)), 0.0)
    return s, int(min(max(round(lo / s), 0), 255)) if s != 1.0 or z else (s, z)


def _affine_no_zero_in_range(x):
    x = np.asarray(x, dtype=np.float64)
    lo, hi = float(x.min()), float(x.max())
    if hi - lo <= 0:
        return 1.0, 0
    s = (hi - lo) / 255
    return s, int(min(max(round(-lo / s), 0), 255))


def _affine_raw_padding(x_real, p):
    v = O.transform_real(np.asarray(x_real, dtype=np.float64), p.hb_in) if p.form == "DH" else np.asarray(x_real)
    s, z = O.affine_params(v)
    q = O.quantize_affine(v, s, z)
    acc = O.conv_codes_wide(q, p.w_int, p.stride, p.pad) - z * p.w_int.astype(np.int64).sum(axis=(1, 2, 3))
    t = (s * p.s_w) * acc.astype(np.float64)
    y = O.transform_real(t, p.hb_out) if p.form == "WH" else t
    y = y + p.bbar if p.form == "DH" else y + O.transform_real(p.bbar, p.hb_out)
    return (np.maximum(y, 0.0) if p.act == "relu" else y), s, z


def _gdn_unsquared(v, beta, gamma, inverse=False):
    v = np.asarray(v, dtype=np.float64)
    norm = np.sqrt(np.asarray(beta, np.float64) + np.abs(v) @ np.asarray(gamma, np.float64).T)
    return v * norm if inverse else v / norm


def _igdn_divides(v, beta, gamma, inverse=False):
    return _orig["gdn"](v, beta, gamma, False)


def _gdn_pool_unsquared(z, g):
    return g.B + np.abs(np.asarray(z, dtype=np.int64)) @ g.G.T


def _gdn_pool_transposed(z, g):
    return g.B + (np.asarray(z, dtype=np.int64) ** 2) @ g.G


def _gdn_int_floor(z, g):
    z = np.asarray(z, dtype=np.int64)
    D = O.gdn_pool(z, g)
    q = (4 * g.P * z * z * D) >> g.t if g.inverse else (4 * g.P * z * z) // (D << g.t)
    return np.sign(z) * np.minimum(127, O.isqrt_floor(np.minimum(q, 255 ** 2)) // 2)


def _order_real_by_sqrt_c(x, m):
    c = np.shape(x)[-1]
    return _orig["transform_order_real"](x, m) * math.sqrt(m) / math.sqrt(c)


def _order_int_transposed(x, m):
    x = np.asarray(x, dtype=np.int64)
    H = _orig["hadamard_of_order"](m)
    return x @ H.T[:x.shape[-1], :]


def _order_quant_sqrt_c(x_i8, m, s_in, s_x):
    x = np.asarray(x_i8, dtype=np.int64)
    rho = float(np.float32(s_in)) / (math.sqrt(x.shape[-1]) * float(np.float32(s_x)))
    M, n = O.fixed_point([rho], [127 * x.shape[-1]], 1)
    y = O.transform_order_int(x, m)
    return np.clip(O.rshift_rne(int(M[0]) * y, n), -127, 127).astype(np.int8)


def _orders_paley2_first(m, orders=None):
    if m == 12:
        return _orig["paley2"](5)
    return _orig["hadamard_of_order"](m, orders)


MUTATIONS = {
    "order_normalized_by_sqrt_c": ("transform_order_real", _order_real_by_sqrt_c),
    "order_transposed": ("transform_order_int", _order_int_transposed),
    "order_paley2_first": ("hadamard_of_order", _orders_paley2_first),
    "order_quantizer_sqrt_c": ("quantize_act_order_i8", _order_quant_sqrt_c),
    "gdn_norm_unsquared": ("gdn", _gdn_unsquared),
    "igdn_divides": ("gdn", _igdn_divides),
    "gdn_pool_unsquared": ("gdn_pool", _gdn_pool_unsquared),
    "gdn_pool_transposed": ("gdn_pool", _gdn_pool_transposed),
    "gdn_int_floor": ("gdn_int", _gdn_int_floor),
    "affine_zero_point_sign": ("affine_params", _affine_z_sign),
    "affine_zero_not_in_range": ("affine_params", _affine_no_zero_in_range),
    "affine_padding_raw_code": ("conv_layer_affine", _affine_raw_padding),
    "convT_forward_gather": ("conv_transpose_codes", _convT_gather),
    "convT_pad_off_by_one": ("conv_transpose_real", _convT_real_unflipped_pad),
    "depth_to_space_channel_order": ("depth_to_space", _d2s_swapped),
    "paley1_identity_dropped": ("paley1", _paley1_no_identity),
    "jacobsthal_chi0": ("_jacobsthal", _jacobsthal_chi0),
    "padded_unnormalized": ("padded_transforms", _padded_unnormalized),
    "general_M_after_H_out": ("epilogue_general", _general_h_before_m),
    "general_lut_index_shift": ("epilogue_general", _general_lut_shifted),
    "phi_sign": ("phi", _phi_sign),
    "profile_non_strict": ("range_expansion_codes", _profile_non_strict),
    "profile_unnormalized": ("range_expansion_codes", _profile_unnormalized),
    "select_non_strict": ("select_form", _select_non_strict),
    "sylvester_sign": ("sylvester", _sylvester_bad),
    "normalize_by_m": ("transform_real", _transform_real_bad),
    "int_transform_sign": ("transform_int", _transform_int_bad),
    "shift_floor": ("rshift_rne", _rshift_floor),
    "fixed_point_gain_dropped": ("fixed_point", _fixed_point_no_gain),
    "gamma_in_dropped": ("prepare_layer", _prepare_no_gamma_in),
    "M_after_H_out": ("epilogue_int", _epilogue_m_after_h),
    "bias_dropped": ("epilogue_int", _epilogue_no_bias),
    "conv_stride_pad_swapped": ("conv_codes", _conv_swap),
    "act_requant_no_sqrt": ("act_multiplier", _act_mult_no_sqrt),
    "wh_transform_wrong_axis": ("transform_weights", _wh_wrong_axis),
    "quantizer_floor": ("quantize_sym", _quantize_floor),
}


def _pins():
    """Every pin test, expanded over its parametrization."""
    out = []
    for name in dir(P):
        if not name.startswith("test_"):
            continue
        fn = getattr(P, name)
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        if not params:
            out.append((name, fn, {}))
            continue
        m = params[0]
        argnames = [a.strip() for a in m.args[0].split(",")] if isinstance(m.args[0], str) else list(m.args[0])
        for vals in m.args[1]:
            vals = vals if len(argnames) > 1 else (vals,)
            out.append((name, fn, dict(zip(argnames, vals))))
    return out


@pytest.mark.parametrize("mutation", sorted(MUTATIONS))
def test_planted_mistake_is_caught(mutation, monkeypatch):
    attr, bad = MUTATIONS[mutation]
    monkeypatch.setattr(O, attr, bad)
    caught = []
    for name, fn, kw in _pins():
        try:
            fn(**kw)
        except (Exception, pytest.fail.Exception):  # a failed pin or an error in the mutated oracle
            caught.append(name)
    assert caught, f"no pin catches the planted mistake {mutation}"
