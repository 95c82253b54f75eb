"""C-ABI checks that need no GPU: the library builds and loads, exports every
function include/hatq.h declares, validates arguments on the host, and its
offline weight preparation (hatq_prepare_weights_host) reproduces the CPU
oracle bit for bit (codes, bias codes, multipliers, shift)."""
import ctypes
import json
import os

import numpy as np
import pytest

from oracle import hatq_oracle as O
from paper_2608_01653_gb300 import hatq as H
from synth import configs as C
from synth import inputs as I

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def lib():
    return H.load()


def test_exports_every_declared_function(lib):
    names = H.declared_functions()
    assert "hatq_conv2d_i8" in names and "hatq_prepare_weights" in names
    assert "hatq_quantize_act" in names and "hatq_layer" in names
    for name in names:
        assert hasattr(lib, name), f"libhatq.so does not export {name}"


def test_selftest_wait_checks_its_limit_on_the_host(lib):
    # argument errors are returned before any launch, so this needs no GPU
    assert lib.hatq_selftest_wait(0, None) == H.ERR_INVALID_ARG
    assert lib.hatq_selftest_wait(4_000_000_001, None) == H.ERR_INVALID_ARG
    assert "limit" in H.last_error()


def test_profile_range_checks_arguments_on_the_host(lib):
    assert lib.hatq_profile_range(None, 0, 4, 4, 64, 64, None, None, None) == H.OK       # empty batch
    assert lib.hatq_profile_range(None, 1, 4, 4, 64, 48, None, None, None) == H.ERR_INVALID_ARG
    assert lib.hatq_profile_range(None, 1, 4, 4, 40, 8, None, None, None) == H.ERR_UNSUPPORTED
    assert lib.hatq_profile_range(None, 1, 4, 4, 64, 64, None, None, None) == H.ERR_INVALID_ARG
    assert "null" in H.last_error()


def test_select_form_decides_exactly(lib):
    """Eq. layerwise_hadamard_selection through the C ABI: WH iff p_l > tau_sel
    (strict), with p_l the exact fraction of expanding images."""
    from fractions import Fraction
    assert H.select_form([1, 1, 1, 1, 0]) == ("DH", Fraction(4, 5))          # p_l = tau_sel: not above it
    assert H.select_form([1] * 5) == ("WH", Fraction(1))
    assert H.select_form([1] * 81 + [0] * 19) == ("WH", Fraction(81, 100))
    assert H.select_form([0, 1], tau=(1, 4)) == ("WH", Fraction(1, 2))
    assert H.select_form([0, 0, 0]) == ("DH", Fraction(0))
    assert H.select_form(np.array([0, 7, 255], np.uint8)) == ("DH", Fraction(2, 3))  # nonzero means expands
    for ind in ([1, 0, 1, 1, 1, 1], [1] * 9 + [0], [0] * 7, [1, 1, 1, 1, 1, 0, 0]):
        form, p = H.select_form(ind)
        assert (form, p) == (O.select_form(O.expansion_probability(ind)), O.expansion_probability(ind))
    for bad in (([], (4, 5)), ([1], (6, 5)), ([1], (1, 0)), ([1], (-1, 5))):
        with pytest.raises(H.HatqError) as e:
            H.select_form(*bad)
        assert e.value.status == H.ERR_INVALID_ARG


class _FakeLayer:
    """The attributes the binding's argument checks read from a prepared layer."""
    c_in, out_f32 = 64, False

    @staticmethod
    def out_shape(n, h, w):
        return (n, h, w, 32)


@pytest.mark.parametrize("call", ["layer", "layer_noalloc", "conv2d_i8"])
def test_binding_rejects_mismatched_tensors_before_the_library(call):
    """Tensors that do not match the layer (channels, dtype for the input kind,
    layout, output shape or dtype) raise ValueError in the binding, before any
    library call could read or write past them."""
    import torch
    L = _FakeLayer()
    fn = getattr(H, call)

    def go(x, kind=H.IN_I8, y=None):
        return fn(x, y=y, L=L) if call == "conv2d_i8" else fn(x, kind, 0.05, L, y=y)
    x8 = torch.zeros((1, 4, 4, 64), dtype=torch.int8)
    with pytest.raises(ValueError, match="channels"):
        go(torch.zeros((1, 4, 4, 48), dtype=torch.int8))
    with pytest.raises(ValueError, match="int8"):
        go(torch.zeros((1, 4, 4, 64), dtype=torch.float16))
    if call != "conv2d_i8":
        with pytest.raises(ValueError, match="float16"):
            go(x8, kind=H.IN_F16)
    with pytest.raises(ValueError, match="contiguous"):
        go(torch.zeros((1, 4, 64, 4), dtype=torch.int8).permute(0, 1, 3, 2))
    with pytest.raises(ValueError, match="shape"):
        go(x8, y=torch.zeros((1, 4, 4, 64), dtype=torch.int8))
    with pytest.raises(ValueError, match="int8"):
        go(x8, y=torch.zeros((1, 4, 4, 32), dtype=torch.float32))
    with pytest.raises(ValueError, match="4-D"):
        go(torch.zeros((4, 4, 64), dtype=torch.int8))
    with pytest.raises(ValueError, match="CUDA"):
        go(x8)


def test_version_and_last_error(lib):
    assert H.version() == 1
    d = H.make_desc(64, 48, 3, 1, 1, "DH", hb_in=64)          # c_out not a multiple of 32
    with pytest.raises(H.HatqError) as e:
        H.prepared_sizes(d)
    assert e.value.status == H.ERR_UNSUPPORTED and "c_out" in H.last_error()


@pytest.mark.parametrize("desc,k_pad", [
    (H.make_desc(192, 192, 5, 2, 2, "DH", hb_in=64), 25 * 192),
    (H.make_desc(3, 192, 5, 2, 2, "WH", hb_out=64), 128),       # small-channel packing 5 x 16 -> 128
    (H.make_desc(3, 64, 3, 1, 1, "WH", hb_out=64), 64),         # 3 x 16 -> 64
    (H.make_desc(5, 64, 5, 1, 2, "WH", hb_out=64), 192),        # 5 x 32 -> 192
    (H.make_desc(32, 224, 3, 1, 1, "DH", hb_in=32), 320),       # c_in % 64 == 32: taps unpadded, 288 -> 320
    (H.make_desc(224, 128, 3, 1, 1, "WH", hb_out=128), 9 * 224 + 32),
    (H.make_desc(96, 64, 1, 1, 0, "DH", hb_in=32), 128),
    (H.make_desc(48, 64, 3, 1, 1, "DH", hb_in=16), 9 * 64),     # c_in % 64 == 48: padded to 64 per tap
    (H.make_desc(128, 128, 1, 1, 0, "DH", hb_in=128), 128),
])
def test_prepared_sizes(desc, k_pad):
    w, c = H.prepared_sizes(desc)
    assert c == desc.c_out and w == desc.c_out * k_pad


@pytest.mark.parametrize("bad", [
    dict(c_in=192, c_out=192, k=5, stride=3, pad=2, form="DH", hb_in=64),     # stride 3
    dict(c_in=192, c_out=192, k=5, stride=2, pad=2, form="DH", hb_in=48),     # block not a power of two
    dict(c_in=192, c_out=192, k=5, stride=2, pad=2, form="DH", hb_in=128),    # block does not divide c_in
    dict(c_in=192, c_out=192, k=5, stride=2, pad=2, form="WH", hb_out=256),   # WH block too large
    dict(c_in=192, c_out=192, k=5, stride=2, pad=5, form="DH", hb_in=64),     # pad >= k
    dict(c_in=3, c_out=192, k=5, stride=2, pad=2, form="DH", hb_in=2),        # DH with c_in % 16
    dict(c_in=192, c_out=192, k=5, stride=2, pad=2, form="XX", hb_in=64),
])
def test_invalid_descriptors_rejected(bad):
    form = {"DH": H.DH, "WH": H.WH}.get(bad.pop("form"), 7)
    d = H.make_desc(form=form, **bad)
    with pytest.raises(H.HatqError) as e:
        H.prepared_sizes(d)
    assert e.value.status in (H.ERR_INVALID_ARG, H.ERR_UNSUPPORTED)


def test_prepare_rejects_bad_scales_and_float_output_with_a_next_transform():
    d = H.make_desc(64, 128, 3, 1, 1, "WH", hb_out=128)
    w = np.zeros((128, 3, 3, 64), np.float32)
    with pytest.raises(H.HatqError):
        H.prepare_weights_host(d, w, None, -1.0, 0.1)
    with pytest.raises(H.HatqError):
        H.prepare_weights_host(d, w, None, 0.1, 0.1, out_f32=True, hb_next=64)


def _oracle_packed(p, desc, k_pad):
    """The oracle's OHWI codes laid out in the library's packed reduction order."""
    co, kh, kw, ci = p.w_int.shape
    out = np.zeros((co, k_pad), np.int8)
    if ci % 16:
        seg = (kw * ci + 7) // 8 * 8            # one kernel row (kx, ci), zero-padded to a multiple of 8
        tmp = np.zeros((co, kh, seg), np.int8)
        tmp[:, :, :kw * ci] = p.w_int.reshape(co, kh, kw * ci)
        out[:, :kh * seg] = tmp.reshape(co, -1)
    else:
        cin_pad = ci if ci % 64 == 32 else (ci + 63) // 64 * 64
        tmp = np.zeros((co, kh * kw, cin_pad), np.int8)
        tmp[:, :, :ci] = p.w_int.reshape(co, kh * kw, ci)
        out[:, :kh * kw * cin_pad] = tmp.reshape(co, -1)
    return out


def _all_layers():
    calib = json.load(open(os.path.join(GOLDEN, "calibration.json")))["configs"]
    for cname in ("cfg0", "cfg1", "cfg2", "cfg3"):
        cfg = C.CONFIGS[cname]
        for ch in cfg.chains:
            plan = C.plan_chain(ch)
            params = C.chain_params(ch)
            for i, L in enumerate(ch.layers):
                last = i == len(ch.layers) - 1
                yield (f"{cname}/{ch.name}/{L.name}", L, params[i], calib[cname][ch.name][i], plan[i],
                       ch.out_f32 and last)


@pytest.mark.parametrize("case", list(_all_layers()), ids=lambda c: c[0])
def test_host_prepare_matches_oracle_bit_exact(case):
    name, L, (w, b), sc, hb_next, out_f32 = case
    desc = H.desc_from_spec(L)
    got = H.prepare_weights_host(desc, w, b, sc["s_x"], sc["s_out"], L.act, hb_next, out_f32)
    ref = O.prepare_layer(w, b, L.form, L.hb_in, L.hb_out, sc["s_x"], sc["s_out"], L.act, hb_next, out_f32,
                          L.stride, L.pad)
    assert np.array_equal(got.w_i8, _oracle_packed(ref, desc, got.w_i8.shape[1]))
    assert np.array_equal(got.w_f16.view(np.float16).astype(np.int64), got.w_i8.astype(np.int64))
    assert np.array_equal(got.b_int, ref.b_int)
    assert np.array_equal(got.s_w, ref.s_w.astype(np.float32))
    if out_f32:
        assert np.array_equal(got.deq, ref.deq.astype(np.float32))
    else:
        assert got.shift == ref.n
        assert np.array_equal(got.mult.astype(np.int64), ref.M)


@pytest.mark.parametrize("L,hb_next", [
    (C.layer("p", 32, 192, 5, 2, 2, "WH", "relu", hb_out=64), 64),     # 25 taps of 32: 800 -> 832
    (C.layer("p", 96, 64, 3, 1, 1, "DH", "none", hb_in=32), 0),        # blocks straddling taps
    (C.layer("p", 160, 128, 1, 1, 0, "DH", "relu", hb_in=32), 128),    # one tap, 160 -> 192
    (C.layer("p", 224, 128, 5, 2, 2, "WH", "relu", hb_out=128), 0),    # 5600 -> 5632, drains
], ids=lambda v: getattr(v, "name", str(v)) if not isinstance(v, int) else str(v))
def test_host_packing_at_32_channel_granularity(L, hb_next):
    """c_in % 64 == 32: the taps follow one another unpadded (k = tap c_in + c),
    the total padded with zero weights to a multiple of 64; codes, bias and
    (M, n) equal the oracle's."""
    w, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=L.c_in), I.bias(L.c_out, seed=L.c_in + 1)
    desc = H.desc_from_spec(L)
    got = H.prepare_weights_host(desc, w, b, 0.05, 0.07, L.act, hb_next, False)
    ref = O.prepare_layer(w, b, L.form, L.hb_in, L.hb_out, 0.05, 0.07, L.act, hb_next, False, L.stride, L.pad)
    k_real = L.k * L.k * L.c_in
    assert got.w_i8.shape[1] == (k_real + 63) // 64 * 64
    assert np.array_equal(got.w_i8[:, :k_real], ref.w_int.reshape(L.c_out, k_real))
    assert not got.w_i8[:, k_real:].any()
    assert np.array_equal(got.b_int, ref.b_int) and got.shift == ref.n
    assert np.array_equal(got.mult.astype(np.int64), ref.M)


def test_host_prepare_zero_weights_and_no_bias():
    d = H.make_desc(64, 64, 1, 1, 0, "DH", hb_in=64)
    w = np.zeros((64, 1, 1, 64), np.float32)
    got = H.prepare_weights_host(d, w, None, 0.1, 0.1)
    assert not got.w_i8.any() and np.all(got.s_w == 1.0) and not got.b_int.any()


def _general_scales(L, w, b, kind, hb_next, seed):
    x_real = np.maximum(I.activations((1, 6, 7, L.c_in), seed=seed).astype(np.float64), 0)
    y = O.conv_real(x_real, w, b, L.stride, L.pad)
    u = np.vectorize(lambda v: O.phi(kind, v))(y)
    s_x = O.symmetric_scale(O.transform_real(x_real, L.hb_in)) if L.form == "DH" else O.symmetric_scale(x_real)
    tgt = O.transform_real(u, hb_next) if hb_next else u
    return (float(np.float32(s_x)), float(np.float32(O.symmetric_scale(y))), float(np.float32(O.symmetric_scale(u))),
            float(np.float32(O.symmetric_scale(tgt))))


GENERAL_CASES = [
    ("dh3x3_silu", C.layer("a", 64, 64, 3, 1, 1, "DH", "silu", hb_in=64), 0),
    ("wh3x3_gelu_next64", C.layer("a", 64, 128, 3, 1, 1, "WH", "gelu", hb_out=64), 64),
    ("dh5x5s2_gelu_next32", C.layer("a", 192, 192, 5, 2, 2, "DH", "gelu", hb_in=64), 32),
    ("wh5x5s2_c3_silu", C.layer("a", 3, 64, 5, 2, 2, "WH", "silu", hb_out=32), 64),
]


@pytest.mark.parametrize("case", GENERAL_CASES, ids=lambda c: c[0])
def test_general_host_prepare_matches_oracle_bit_exact(case):
    name, L, hb_next = case
    w = I.weights(L.c_out, L.k, L.k, L.c_in, seed=31)
    b = I.bias(L.c_out, seed=32)
    s_x, s_z, s_u, s_y = _general_scales(L, w, b, L.act, hb_next, 33)
    got = H.prepare_weights_general_host(H.desc_from_spec(L), w, b, s_x, s_z, s_u, s_y, L.act, hb_next)
    ref = O.prepare_layer(w, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, False, L.stride, L.pad,
                          s_z=s_z, s_u=s_u)
    assert np.array_equal(got.w_i8, _oracle_packed(ref, H.desc_from_spec(L), got.w_i8.shape[1]))
    assert np.array_equal(got.b_int, ref.b_int)
    assert np.array_equal(got.mult.astype(np.int64), ref.M) and got.shift == ref.n
    assert got.mult_in == ref.M_in and got.shift_in == ref.n_in
    assert np.array_equal(got.lut[:255].astype(np.int64), ref.lut)


def test_general_prepare_rejects_what_it_does_not_cover(lib):
    d = H.make_desc(64, 128, 3, 1, 1, "WH", hb_out=128)
    w = np.zeros((128, 3, 3, 64), np.float32)
    with pytest.raises(H.HatqError) as e:                       # 128-wide output block
        H.prepare_weights_general_host(d, w, None, 0.1, 0.1, 0.1, 0.1, "silu", 0)
    assert e.value.status == H.ERR_UNSUPPORTED
    d = H.make_desc(64, 64, 3, 1, 1, "DH", hb_in=64)
    w = np.zeros((64, 3, 3, 64), np.float32)
    with pytest.raises(H.HatqError) as e:                       # nonpositive activation scale
        H.prepare_weights_general_host(d, w, None, 0.1, 0.0, 0.1, 0.1, "gelu", 0)
    assert e.value.status == H.ERR_INVALID_ARG
    with pytest.raises(H.HatqError) as e:                       # SiLU through the homogeneous entry point
        H.prepare_weights_host(d, w, None, 0.1, 0.1, "silu", 0)
    assert e.value.status == H.ERR_INVALID_ARG


def test_binding_constants_match_the_header():
    """The Python binding's status, form, activation and input-kind values
    are the ones include/hatq.h declares."""
    import re
    text = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "hatq.h")).read()
    decl = {k: int(v) for k, v in re.findall(r"\b(HATQ_[A-Z0-9_]+)\s*=\s*(\d+)", text)}
    expect = {"HATQ_OK": H.OK, "HATQ_ERR_INVALID_ARG": H.ERR_INVALID_ARG, "HATQ_ERR_UNSUPPORTED": H.ERR_UNSUPPORTED,
              "HATQ_ERR_OVERFLOW": H.ERR_OVERFLOW, "HATQ_ERR_CUDA": H.ERR_CUDA, "HATQ_ERR_TIMEOUT": H.ERR_TIMEOUT,
              "HATQ_DH": H.DH, "HATQ_WH": H.WH, "HATQ_ACT_NONE": H.ACT_NONE, "HATQ_ACT_RELU": H.ACT_RELU,
              "HATQ_ACT_SILU": H.ACT_SILU, "HATQ_ACT_GELU": H.ACT_GELU, "HATQ_IN_OPERAND": H.IN_OPERAND,
              "HATQ_IN_I8": H.IN_I8, "HATQ_IN_F16": H.IN_F16}
    for name, value in expect.items():
        assert decl[name] == value, name
    m = re.search(r"#define\s+HATQ_NOALLOC_MAX_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", text)
    assert m and (int(m.group(1)) << int(m.group(2))) == H.NOALLOC_MAX_BYTES


def test_prepared_struct_mirror_matches_the_c_layout(tmp_path):
    """The ctypes mirror of hatq_prepared has the size and field offsets the C
    compiler gives the header's struct (the library writes the whole struct)."""
    import ctypes
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    fields = ["d", "act", "hb_next", "out_f32", "shift", "k_pad", "gather", "s_x", "s_y", "w_i8", "w_f16", "b_int",
              "mult", "deq", "s_w", "opaque", "s_z", "s_u", "shift_in", "in_affine", "mult_in", "lut"]
    src = tmp_path / "layout.c"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    src.write_text("#include <stdio.h>\n#include <stddef.h>\n#include \"hatq.h\"\nint main(void) {\n"
                   "  printf(\"%zu\\n\", sizeof(hatq_prepared));\n"
                   + "".join(f"  printf(\"%zu\\n\", offsetof(hatq_prepared, {f}));\n" for f in fields)
                   + "  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", inc, str(src), "-o", str(exe)], check=True, capture_output=True)
    out = [int(v) for v in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert ctypes.sizeof(H.PreparedStruct) == out[0]
    for f, off in zip(fields, out[1:]):
        assert getattr(H.PreparedStruct, f).offset == off, f


@pytest.mark.parametrize("hb_out", [0, 16, 32, 64, 128])
def test_every_transition_block_pair_is_accepted(hb_out):
    """Every WH output block and next-layer DH input block of Table
    integer_transitions up to 128 is one fused transition in the library
    (the paper's single requantization, Eq. integer_hadamard_transition)."""
    c = 128
    d = H.make_desc(64, c, 1, 1, 0, "WH", hb_out=hb_out) if hb_out else H.make_desc(64, c, 1, 1, 0, "DH", hb_in=64)
    w = np.zeros((c, 1, 1, 64), np.float32)
    w[:, 0, 0, 0] = 0.5
    for hb_next in (0, 16, 32, 64, 128):
        got = H.prepare_weights_host(d, w, None, 0.1, 0.1, "relu", hb_next)
        ref = O.prepare_layer(w, None, "WH" if hb_out else "DH", 0 if hb_out else 64, hb_out, 0.1, 0.1, "relu",
                              hb_next, False, 1, 0)
        assert got.shift == ref.n and np.array_equal(got.mult.astype(np.int64), ref.M), (hb_out, hb_next)


def test_chain_plan_is_the_oracles_transition_plan():
    """The CUDA path's chain planner (synth.configs.plan_chain) and the
    oracle's own reading of Table integer_transitions agree on every chain."""
    for cfg in C.CONFIGS.values():
        for ch in cfg.chains:
            assert C.plan_chain(ch) == O.transition_blocks(ch.layers), ch.name


# ------------------------------------------------------------------ the paper's single order (f2)

def test_library_orders_and_matrices_match_the_oracle():
    """The library builds the same M_H, m(C) and H~_m as the oracle (two
    independent implementations of the supplementary's constructions under
    the same choice rule)."""
    for c in range(1, 700):
        assert H.hadamard_order(c) == O.hadamard_order(c), c
    orders = O.supported_orders(1024)
    for m in [k for k in sorted(orders) if k <= 512] + [576, 640, 768, 1024]:
        assert np.array_equal(H.hadamard_matrix(m).astype(np.int64), O.hadamard_of_order(m, orders)), m
    with pytest.raises(H.HatqError):
        H.hadamard_matrix(100)                     # not in M_H (Paley needs a prime q)


ORDER_CASES = [
    ("dh5x5s2_c192_m192", C.layer("a", 192, 192, 5, 2, 2, "DH", "relu", hb_in=64), 0),
    ("dh3x3_c190_m192_pad", C.layer("a", 190, 64, 3, 1, 1, "DH", "none", hb_in=2), 0),
    ("dh3x3_c320_m320_kron", C.layer("a", 320, 640, 3, 1, 1, "DH", "relu", hb_in=64), 128),
    ("dh3x3_c224_m224_next32", C.layer("a", 224, 128, 3, 1, 1, "DH", "relu", hb_in=32), 32),
]


@pytest.mark.parametrize("case", ORDER_CASES, ids=lambda c: c[0])
def test_order_host_prepare_matches_oracle_bit_exact(case):
    name, L, hb_next = case
    m = O.hadamard_order(L.c_in)
    w, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=61), I.bias(L.c_out, seed=62)
    desc = H.make_desc(L.c_in, L.c_out, L.k, L.stride, L.pad, "DH")
    got = H.prepare_weights_order_host(desc, w, b, 0.07, 0.05, L.act, hb_next)
    ref = O.prepare_layer(w, b, "DH", 0, 0, 0.07, 0.05, L.act, hb_next, False, L.stride, L.pad, order_in=m)
    dop = H.order_desc(desc)
    assert dop.c_in == m and dop.hb_in == m
    assert np.array_equal(got.w_i8, _oracle_packed(ref, dop, got.w_i8.shape[1]))
    assert np.array_equal(got.b_int, ref.b_int)
    assert got.shift == ref.n and np.array_equal(got.mult.astype(np.int64), ref.M)


def test_order_layers_reject_what_they_do_not_cover(lib):
    w = np.zeros((64, 3, 3, 192), np.float32)
    with pytest.raises(H.HatqError) as e:          # a block prepare with a non-power-of-two block
        H.prepare_weights_host(H.make_desc(192, 64, 3, 1, 1, "DH", hb_in=192), w, None, 0.1, 0.1)
    assert e.value.status == H.ERR_INVALID_ARG
    with pytest.raises(H.HatqError) as e:          # the single order is built for DH layers
        H.prepare_weights_order_host(H.make_desc(192, 64, 3, 1, 1, "WH", hb_out=64), w, None, 0.1, 0.1)
    assert e.value.status == H.ERR_UNSUPPORTED
    w_elems, ch = H.prepared_sizes(H.ConvDesc(190, 192, 1, 1, 1, 0, H.TRANSFORM, 0, 0))
    assert ch == 192 and w_elems == 192 * 192      # 1x1 with c = 190 -> packed reduction 192
    for bad in (H.ConvDesc(192, 192, 3, 3, 1, 1, H.TRANSFORM, 0, 0), H.ConvDesc(192, 100, 1, 1, 1, 0, H.TRANSFORM, 0, 0)):
        with pytest.raises(H.HatqError):
            H.prepared_sizes(bad)


def test_transposed_struct_mirror_matches_the_c_layout(tmp_path):
    """The ctypes mirror of hatq_prepared_transposed has the C layout."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    fields = ["d", "out_pad", "classes", "pad_y", "pad_x", "sub"]
    src = tmp_path / "tlayout.c"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    src.write_text("#include <stdio.h>\n#include <stddef.h>\n#include \"hatq.h\"\nint main(void) {\n"
                   "  printf(\"%zu\\n\", sizeof(hatq_prepared_transposed));\n"
                   + "".join(f"  printf(\"%zu\\n\", offsetof(hatq_prepared_transposed, {f}));\n" for f in fields)
                   + "  return 0;\n}\n")
    exe = tmp_path / "tlayout"
    subprocess.run([cc, "-I", inc, str(src), "-o", str(exe)], check=True, capture_output=True)
    out = [int(v) for v in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert ctypes.sizeof(H.PreparedTransposedStruct) == out[0]
    for f, off in zip(fields, out[1:]):
        assert getattr(H.PreparedTransposedStruct, f).offset == off, f


@pytest.mark.parametrize("k,s,p,cls,taps", [(5, 2, 2, 0, (3, 3)), (5, 2, 2, 3, (2, 2)), (4, 2, 1, 1, (2, 2)),
                                            (3, 2, 1, 2, (2, 1)), (3, 1, 1, 0, (3, 3))])
def test_transposed_class_sizes(k, s, p, cls, taps):
    """Class (py, px) of a transposed convolution is a stride-1 sub-convolution
    with the taps ky = py + p (mod s), kx likewise."""
    d = H.make_desc(64, 128, k, s, p, "DH", hb_in=64)
    w, c = ctypes.c_size_t(), ctypes.c_size_t()
    assert H.load().hatq_transposed_sizes(ctypes.byref(d), cls, ctypes.byref(w), ctypes.byref(c)) == H.OK
    assert c.value == 128 and w.value == 128 * taps[0] * taps[1] * 64
    assert H.load().hatq_transposed_sizes(ctypes.byref(d), s * s, ctypes.byref(w), ctypes.byref(c)) == H.ERR_INVALID_ARG


# ------------------------------------------------ GDN / IGDN (integer phi_int, reading R21)

def _gdn_inputs(c, seed, scale=0.01):
    rng = np.random.default_rng(seed)
    beta = 0.5 + rng.random(c)
    gamma = np.abs(rng.standard_normal((c, c))) * scale
    return beta, gamma


@pytest.mark.parametrize("c,inverse,hb_next", [(64, False, 0), (128, True, 64), (192, False, 16), (256, True, 1),
                                               (192, True, 32)])
def test_prepare_gdn_host_matches_oracle(lib, c, inverse, hb_next):
    """The library's pool coefficients, pool bias, scale exponent, fixed-point
    R^2 and input-side (M_in, n_in) equal the oracle's (R21 and R3)."""
    beta, gamma = _gdn_inputs(c, c + int(inverse))
    s_z, s_u, s_y = 0.043, 0.021 if not inverse else 0.09, 0.05
    h = H.prepare_gdn_host(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next)
    g = O.gdn_params(beta, gamma, s_z, s_u, inverse)
    assert np.array_equal(h.G, g.G) and np.array_equal(h.B, g.B)
    assert (h.e, h.P, h.t) == (g.e, g.P, g.t)
    g_in = np.sqrt(hb_next) if hb_next else 1.0
    M, n = O.fixed_point([float(np.float32(s_u)) / (g_in * float(np.float32(s_y)))], [127], hb_next if hb_next else 1)
    assert (h.mult_in, h.shift_in) == (int(M[0]), n)


def test_gdn_preactivation_layer_is_a_plain_layer():
    """The GPU runs GDN as a plain layer (act none, output scale s_z) followed
    by hatq_gdn: its (M, n) equal the general transition's (M_out, n_out)."""
    w, b = I.weights(64, 3, 3, 64, seed=5), I.bias(64, seed=6)
    beta, gamma = _gdn_inputs(64, 1)
    pg = O.prepare_layer(w, b, "DH", 64, 0, 0.02, 0.05, "gdn", 0, False, 1, 1, s_z=0.03, s_u=0.04,
                         gdn_beta=beta, gdn_gamma=gamma)
    pp = O.prepare_layer(w, b, "DH", 64, 0, 0.02, 0.03, "none", 0, False, 1, 1)
    assert np.array_equal(pg.M, pp.M) and pg.n == pp.n


def test_prepare_gdn_rejects_on_the_host(lib):
    beta, gamma = _gdn_inputs(64, 2)
    with pytest.raises(H.HatqError) as e:
        H.prepare_gdn_host(96, np.ones(96), np.zeros((96, 96)), 0.1, 0.1, False, 0.1)
    assert e.value.status == H.ERR_UNSUPPORTED
    with pytest.raises(H.HatqError) as e:
        H.prepare_gdn_host(64, beta, gamma, 0.1, 0.1, False, 0.1, hb_next=128)
    assert e.value.status == H.ERR_UNSUPPORTED
    bad = beta.copy()
    bad[3] = 0.0
    with pytest.raises(H.HatqError) as e:
        H.prepare_gdn_host(64, bad, gamma, 0.1, 0.1, False, 0.1)
    assert e.value.status == H.ERR_INVALID_ARG
    with pytest.raises(H.HatqError) as e:
        H.prepare_gdn_host(64, beta, -gamma - 1.0, 0.1, 0.1, False, 0.1)
    assert e.value.status == H.ERR_INVALID_ARG
    with pytest.raises(ValueError):
        H.prepare_gdn_host(64, beta[:10], gamma, 0.1, 0.1, False, 0.1)
    assert lib.hatq_gdn(None, 1, 1, 1, None, None, None) == H.ERR_INVALID_ARG


def test_set_operand_format_checks_on_the_host(lib):
    """hatq_set_operand_format is host-only: it validates the layer kind and
    writes the two flags (no device buffers are touched)."""
    P = H.PreparedStruct()
    P.d = H.make_desc(192, 192, 3, 1, 1, "DH", hb_in=64)
    assert lib.hatq_set_operand_format(ctypes.byref(P), 1, 1) == H.OK and (P.in_f16, P.out_f16) == (1, 1)
    assert lib.hatq_set_operand_format(ctypes.byref(P), 0, 0) == H.OK and (P.in_f16, P.out_f16) == (0, 0)
    assert lib.hatq_set_operand_format(ctypes.byref(P), 2, 0) == H.ERR_INVALID_ARG
    P.gather = 1
    assert lib.hatq_set_operand_format(ctypes.byref(P), 1, 0) == H.ERR_UNSUPPORTED
    P.gather, P.in_affine = 0, 1
    assert lib.hatq_set_operand_format(ctypes.byref(P), 1, 0) == H.ERR_UNSUPPORTED
    P.in_affine, P.out_f32 = 0, 1
    assert lib.hatq_set_operand_format(ctypes.byref(P), 0, 1) == H.ERR_UNSUPPORTED
    P.out_f32 = 0
    P.d = H.make_desc(224, 128, 3, 1, 1, "DH", hb_in=32)      # taps packed at 32-channel granularity
    assert lib.hatq_set_operand_format(ctypes.byref(P), 1, 0) == H.ERR_UNSUPPORTED
    assert lib.hatq_set_operand_format(ctypes.byref(P), 0, 1) == H.OK
    assert lib.hatq_set_operand_format(None, 0, 0) == H.ERR_INVALID_ARG

