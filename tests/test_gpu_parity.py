"""GPU parity: libhatq (through its C ABI) against the CPU oracle on the same
seeded inputs. Integer paths must be bit-exact; the FP16 entry path may
differ by at most one code step on at most 0.1% of codes, with the float
output within relative L2 error 1e-3."""
import json
import os
import zlib

import numpy as np
import pytest

from oracle import hatq_oracle as O
from synth import configs as C
from synth import inputs as I

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
CALIB = json.load(open(os.path.join(GOLDEN, "calibration.json")))["configs"]


@pytest.fixture(scope="module")
def H():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_01653_gb300 import hatq
    hatq.load()
    return hatq


def dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.cpu().numpy()


def assert_codes_close(got, ref, max_frac=1e-3):
    d = np.abs(got.astype(np.int64) - ref.astype(np.int64))
    assert d.max() <= 1, f"max code difference {d.max()}"
    assert np.mean(d > 0) <= max_frac, f"{np.mean(d > 0):.2e} of codes differ"


def rel_l2(got, ref):
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.linalg.norm(np.asarray(got, np.float64) - ref) / max(np.linalg.norm(ref), 1e-300))


# ------------------------------------------------------------------ quantize (a2)

@pytest.mark.parametrize("shape,hb", [((2, 7, 9, 192), 64), ((1, 5, 3, 256), 256), ((1, 4, 4, 128), 128),
                                      ((3, 3, 5, 32), 32), ((1, 6, 7, 16), 16), ((1, 2, 3, 48), 1),
                                      ((1, 9, 1, 64), 2), ((1, 3, 3, 64), 8)])
def test_quantize_i8_static_bit_exact(H, shape, hb):
    x = I.activations_i8(shape, seed=100 + hb, s_in=0.05)
    s_x = 0.05 * np.sqrt(hb) / 3.0
    y = H.quantize_act(dev(x), H.IN_I8, 0.05, hb, s_x)
    H.sync_status()
    ref = O.quantize_act_i8(x, hb, 0.05, s_x)
    assert np.array_equal(host(y), ref)


# (shape, hb, s_in, rho = s_in / (sqrt(hb) s_x)): rho <= 1 takes the packed
# 16-bit-pair kernel; rho = 1/4 at hb = 64 gives M = 2^(n-2), where rounding
# ties occur; rho = 1 gives M = 2^n; odd totals leave a lane half-empty;
# 4096 codes are exactly one warp tile, 4160 one tile and a 64-code tail.
PACKED = [((2, 37, 41, 192), 64, 0.05, 0.3), ((1, 4, 6, 64), 64, 0.5, 0.25), ((1, 5, 5, 64), 64, 0.5, 1.0),
          ((1, 1, 3, 48), 16, 0.05, 0.7), ((1, 1, 5, 16), 16, 0.05, 0.9), ((1, 3, 7, 96), 32, 0.05, 0.05),
          ((1, 2, 9, 48), 1, 0.05, 0.9), ((1, 6, 7, 64), 2, 0.05, 0.5), ((3, 3, 5, 32), 8, 0.05, 0.4),
          ((1, 7, 3, 128), 4, 0.05, 0.6), ((1, 8, 8, 64), 64, 0.05, 0.3), ((1, 1, 65, 64), 64, 0.05, 0.3)]


@pytest.mark.parametrize("shape,hb,s_in,rho", PACKED)
def test_quantize_i8_packed_pairs_bit_exact(H, shape, hb, s_in, rho):
    x = I.activations_i8(shape, seed=400 + hb, s_in=s_in)
    x.reshape(-1)[: min(64, x.size)] = 127                 # coherent blocks: |y| = 127 hb, saturating codes
    s_x = float(np.float32(s_in / (np.sqrt(hb) * rho)))
    y = H.quantize_act(dev(x), H.IN_I8, s_in, hb, s_x)
    H.sync_status()
    ref = O.quantize_act_i8(x, hb, s_in, s_x)
    assert np.array_equal(host(y), ref)
    if rho * hb >= 1:                                       # the coherent block's code rho 127 hb saturates
        assert (np.abs(ref.astype(int)) == 127).any()


@pytest.mark.parametrize("shape,hb", [((1, 16, 16, 128), 128), ((2, 5, 7, 192), 64), ((1, 3, 3, 256), 256),
                                      ((1, 4, 5, 32), 16), ((1, 1, 65, 64), 64), ((3, 7, 5, 32), 32),
                                      ((1, 2, 9, 48), 1), ((2, 9, 11, 64), 2), ((1, 8, 8, 64), 8)])
def test_quantize_f16_static_within_tolerance(H, shape, hb):
    x = I.activations_f16(shape, seed=200 + hb)
    y_real = O.transform_real(x.astype(np.float64), hb)
    s_x = float(np.float32(O.symmetric_scale(y_real)))
    y = H.quantize_act(dev(x), H.IN_F16, 1.0, hb, s_x)
    H.sync_status()
    assert_codes_close(host(y), O.quantize_act_f16(x, hb, s_x))


@pytest.mark.parametrize("hb", [1, 64, 128])
def test_quantize_i8_dynamic(H, hb):
    x = I.activations_i8((1, 11, 13, 128), seed=300 + hb, s_in=0.05)
    y, s_used = H.quantize_act(dev(x), H.IN_I8, 0.05, hb, 0.0)
    H.sync_status()
    ref, s_ref = O.quantize_act_dynamic_i8(x, hb, 0.05)
    assert np.array_equal(host(y), ref)
    assert float(host(s_used)[0]) == np.float32(s_ref)


@pytest.mark.parametrize("shape,hb", [((2, 37, 41, 192), 64), ((1, 9, 7, 64), 2), ((1, 5, 11, 96), 32),
                                      ((1, 3, 3, 48), 1), ((1, 4, 4, 64), 8), ((1, 1, 65, 64), 64)])
def test_quantize_i8_dynamic_packed_pairs(H, shape, hb):
    """Dynamic scale through the packed-pair max-abs and quantize passes (the
    parameter block selects the packed pass on the device)."""
    x = I.activations_i8(shape, seed=500 + hb, s_in=0.05)
    y, s_used = H.quantize_act(dev(x), H.IN_I8, 0.05, hb, 0.0)
    H.sync_status()
    ref, s_ref = O.quantize_act_dynamic_i8(x, hb, 0.05)
    assert np.array_equal(host(y), ref)
    assert float(host(s_used)[0]) == np.float32(s_ref)
    assert (np.abs(ref.astype(int)) == 127).any()


def test_quantize_i8_dynamic_general_fallback(H):
    """Codes in [-1, 1]: max |y| < 127 gives M > 2^n, so the parameter block
    leaves the quantize pass to the general kernel."""
    x = np.random.default_rng(6).integers(-1, 2, (1, 7, 9, 64)).astype(np.int8)
    y, s_used = H.quantize_act(dev(x), H.IN_I8, 0.05, 4, 0.0)
    H.sync_status()
    ref, s_ref = O.quantize_act_dynamic_i8(x, 4, 0.05)
    assert np.array_equal(host(y), ref)
    assert float(host(s_used)[0]) == np.float32(s_ref)


@pytest.mark.parametrize("shape,hb", [((2, 5, 7, 192), 64), ((1, 3, 3, 48), 16), ((1, 1, 65, 64), 64), ((1, 6, 7, 64), 1)])
def test_quantize_f16_dynamic_wide(H, shape, hb):
    """FP16 entry, dynamic scale, blocks <= 64: the lane-per-block max-abs and
    quantize passes."""
    x = I.activations_f16(shape, seed=700 + hb)
    y, s_used = H.quantize_act(dev(x), H.IN_F16, 1.0, hb, 0.0)
    H.sync_status()
    ref, s_ref = O.quantize_act_dynamic_f16(x, hb)
    assert_codes_close(host(y), ref)
    assert abs(float(host(s_used)[0]) - s_ref) <= 1e-6 * s_ref


def test_quantize_f16_dynamic(H):
    x = I.activations_f16((1, 16, 16, 128), seed=0)
    y, s_used = H.quantize_act(dev(x), H.IN_F16, 1.0, 128, 0.0)
    H.sync_status()
    ref, s_ref = O.quantize_act_dynamic_f16(x, 128)
    assert_codes_close(host(y), ref)
    assert abs(float(host(s_used)[0]) - s_ref) <= 1e-6 * s_ref


def test_quantize_zero_and_empty(H):
    import torch
    x = np.zeros((1, 4, 4, 64), np.int8)
    y, s_used = H.quantize_act(dev(x), H.IN_I8, 0.05, 64, 0.0)
    H.sync_status()
    assert not host(y).any() and float(host(s_used)[0]) == 1.0
    e = torch.zeros((0, 4, 4, 64), dtype=torch.int8, device="cuda")
    assert H.quantize_act(e, H.IN_I8, 0.05, 64, 0.1).numel() == 0


def test_quantize_full_cfg1_input(H):
    ch = C.CONFIGS["cfg1"].chains[0]
    x = C.chain_input(ch)
    s_x = CALIB["cfg1"][ch.name][0]["s_x"]
    y = H.quantize_act(dev(x), H.IN_I8, ch.s_in, 64, s_x)
    H.sync_status()
    assert np.array_equal(host(y), O.quantize_act_i8(x, 64, ch.s_in, s_x))


# ------------------------------------------------------------------ conv + epilogue (a3, a4)

def run_layer(H, L, w, b, s_x, s_y, hb_next, out_f32, x, x_kind, s_in):
    P = H.prepare_weights(H.desc_from_spec(L), w, b, s_x, s_y, L.act, hb_next, out_f32)
    y = H.layer(dev(x), x_kind, s_in, P)
    H.sync_status()
    ref_p = O.prepare_layer(w, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, out_f32, L.stride, L.pad)
    kind = {H.IN_OPERAND: "operand", H.IN_I8: "i8", H.IN_F16: "f16"}[x_kind]
    op = O.layer_operand(x, kind, s_in, L.form, L.hb_in, s_x)
    return host(y), O.conv_layer(op, ref_p), op


def calibrated(L, w, b, x_real, hb_next):
    """Scales from the real-valued model for a single test layer."""
    if L.form == "DH":
        s_x = O.symmetric_scale(O.transform_real(x_real, L.hb_in))
    else:
        s_x = O.symmetric_scale(x_real)
    y = O.conv_real(x_real, w, b, L.stride, L.pad)
    y = np.maximum(y, 0) if L.act == "relu" else y
    s_y = O.symmetric_scale(O.transform_real(y, hb_next) if hb_next else y)
    return float(np.float32(s_x)), float(np.float32(s_y))


LAYER_CASES = [
    # name, layer, input shape (n, h, w), hb_next
    ("dh1x1_k128_nodrain", C.layer("a", 128, 128, 1, 1, 0, "DH", "none", hb_in=128), (1, 16, 16), 0),
    ("dh3x3_k1728_drain", C.layer("a", 192, 192, 3, 1, 1, "DH", "relu", hb_in=64), (2, 13, 37), 64),
    ("dh5x5s2_ragged", C.layer("a", 192, 192, 5, 2, 2, "DH", "none", hb_in=64), (3, 19, 45), 0),
    ("wh5x5s2_c3_gather", C.layer("a", 3, 192, 5, 2, 2, "WH", "relu", hb_out=64), (1, 40, 50), 64),
    ("wh3x3_hb128_split", C.layer("a", 224, 128, 3, 1, 1, "WH", "relu", hb_out=128), (1, 12, 20), 0),
    ("dh3x3_c32_box", C.layer("a", 32, 224, 3, 1, 1, "DH", "relu", hb_in=32), (2, 9, 17), 0),
    ("dh3x3_next128_split", C.layer("a", 128, 128, 3, 1, 1, "DH", "relu", hb_in=128), (1, 10, 33), 128),
    ("dh3x3_c640_n160", C.layer("a", 320, 640, 3, 1, 1, "DH", "relu", hb_in=64), (1, 6, 9), 0),
    ("wh1x1_c640", C.layer("a", 640, 640, 1, 1, 0, "WH", "none", hb_out=128), (1, 7, 11), 0),
    ("dh3x3_next32", C.layer("a", 224, 128, 3, 1, 1, "DH", "relu", hb_in=32), (1, 8, 8), 32),
    ("wh3x3_fused_16", C.layer("a", 64, 64, 3, 2, 1, "WH", "relu", hb_out=16), (1, 16, 24), 16),
    # WH-to-DH transitions with a 128-wide transform on either side (Table integer_transitions):
    # one requantization, the two epilogue warpgroups exchanging halves for the next transform
    ("wh3x3_128_next128_drain", C.layer("a", 224, 128, 3, 1, 1, "WH", "relu", hb_out=128), (2, 11, 21), 128),
    ("wh1x1_128_next128_nodrain", C.layer("a", 128, 128, 1, 1, 0, "WH", "relu", hb_out=128), (1, 13, 29), 128),
    ("wh3x3_128_next64", C.layer("a", 64, 128, 3, 1, 1, "WH", "relu", hb_out=128), (1, 9, 14), 64),
    ("wh3x3_64_next128", C.layer("a", 64, 128, 3, 1, 1, "WH", "relu", hb_out=64), (1, 9, 14), 128),
    ("wh3x3_32_next128", C.layer("a", 96, 128, 3, 2, 1, "WH", "relu", hb_out=32), (1, 17, 23), 128),
    ("dh1x1_next128_nodrain", C.layer("a", 64, 128, 1, 1, 0, "DH", "relu", hb_in=64), (1, 12, 12), 128),
    ("wh3x3_c640_128_next128", C.layer("a", 320, 640, 3, 1, 1, "WH", "relu", hb_out=128), (1, 7, 10), 128),
    ("wh5x5s2_c3_next128", C.layer("a", 3, 128, 5, 2, 2, "WH", "relu", hb_out=128), (1, 30, 44), 128),
    # small-channel layers whose input rows are 16-byte multiples: the window comes by TMA
    ("wh5x5s2_c3_tma_window", C.layer("a", 3, 192, 5, 2, 2, "WH", "relu", hb_out=64), (2, 41, 64), 64),
    ("wh3x3_c4_tma_window", C.layer("a", 4, 64, 3, 1, 1, "WH", "relu", hb_out=64), (1, 21, 36), 0),
    ("wh7x7_c8_tma_window", C.layer("a", 8, 64, 7, 1, 3, "WH", "none", hb_out=32), (2, 19, 34), 32),
    # c_in % 64 == 32: taps packed at 32-channel granularity, two 32-channel boxes per 64-wide block
    # (blocks straddling two taps, a last block half past the last tap, drains)
    ("dh5x5s2_c160_pieces_drain", C.layer("a", 160, 128, 5, 2, 2, "DH", "relu", hb_in=32), (1, 21, 30), 0),
    ("dh1x1_c32_pieces", C.layer("a", 32, 64, 1, 1, 0, "DH", "none", hb_in=32), (2, 7, 13), 0),
    ("wh5x5s2_c32_pieces_next64", C.layer("a", 32, 192, 5, 2, 2, "WH", "relu", hb_out=64), (1, 19, 26), 64),
]


@pytest.mark.parametrize("case", LAYER_CASES, ids=lambda c: c[0])
def test_layer_i8_bit_exact(H, case):
    name, L, (n, h, w), hb_next = case
    x = I.activations_i8((n, h, w, L.c_in), seed=zlib.crc32(name.encode()) % 1000, s_in=0.05)
    wts = I.weights(L.c_out, L.k, L.k, L.c_in, seed=7)
    b = I.bias(L.c_out, seed=8)
    x_real = x.astype(np.float64) * float(np.float32(0.05))
    s_x, s_y = calibrated(L, wts, b, x_real, hb_next)
    if L.form == "WH":
        s_x = 0.05          # WH consumes the INT8 input as is
    got, ref, _ = run_layer(H, L, wts, b, s_x, s_y, hb_next, False, x, H.IN_I8, 0.05)
    assert got.dtype == np.int8
    assert np.array_equal(got, ref)
    assert np.mean(np.abs(ref.astype(int)) == 127) < 0.2      # not a saturated comparison


@pytest.mark.parametrize("case", [c for c in LAYER_CASES if c[3] == 0], ids=lambda c: c[0])
def test_layer_f32_output(H, case):
    name, L, (n, h, w), _ = case
    x = I.activations_i8((n, h, w, L.c_in), seed=11, s_in=0.05)
    wts = I.weights(L.c_out, L.k, L.k, L.c_in, seed=12)
    b = I.bias(L.c_out, seed=13)
    s_x, _ = calibrated(L, wts, b, x.astype(np.float64) * 0.05, 0)
    if L.form == "WH":
        s_x = 0.05
    got, ref, _ = run_layer(H, L, wts, b, s_x, 1.0, 0, True, x, H.IN_I8, 0.05)
    assert got.dtype == np.float32
    assert rel_l2(got, ref) <= 1e-5


def _spike_weights(co, k, ci, hb):
    """Weights whose DH transform is flat: every transformed code is +127."""
    w = np.zeros((co, k, k, ci), np.float32)
    w[..., ::hb] = 1.0
    return w


@pytest.mark.parametrize("sign", [1, -1])
def test_accumulator_exact_beyond_fp32_integer_range(H, sign):
    """|sum| = 127^2 * 4800 > 2^24 at interior pixels; a bias cancels it so the
    INT8 output shows the accumulator's low bits (M / 2^n = 1)."""
    L = C.layer("a", 192, 64, 5, 1, 2, "DH", "none", hb_in=64)
    w = _spike_weights(64, 5, 192, 64)
    x = np.full((1, 12, 12, 192), 127 * sign, np.int8)
    s_x = 0.01
    s_w = float(1.0 / np.sqrt(64) / 127)
    full = 127 * 127 * 25 * 192
    b = np.full(64, -sign * (full - 3) * s_x * s_w, np.float32)
    b[1::2] = -sign * (full + 40) * s_x * s_w
    s_y = float(np.float32(s_x * s_w))
    got, ref, _ = run_layer(H, L, w, b, s_x, s_y, 0, False, x, H.IN_OPERAND, s_x)
    assert np.array_equal(got, ref)
    interior = ref[0, 2:-2, 2:-2, :].astype(np.int64)
    assert np.all(np.abs(interior) < 127) and len(np.unique(interior)) >= 2


def test_cfg0_fp16_entry(H):
    ch = C.CONFIGS["cfg0"].chains[0]
    L = ch.layers[0]
    x = C.chain_input(ch)
    (w, b), = C.chain_params(ch)
    sc = CALIB["cfg0"][ch.name][0]
    got, ref, op = run_layer(H, L, w, b, sc["s_x"], sc["s_out"], 0, True, x, H.IN_F16, 1.0)
    assert rel_l2(got, ref) <= 1e-3
    y = H.quantize_act(dev(x), H.IN_F16, 1.0, L.hb_in, sc["s_x"])
    H.sync_status()
    assert_codes_close(host(y), op)


def test_cfg1_full_bit_exact(H):
    ch = C.CONFIGS["cfg1"].chains[0]
    L = ch.layers[0]
    x = C.chain_input(ch)
    (w, b), = C.chain_params(ch)
    sc = CALIB["cfg1"][ch.name][0]
    got, ref, _ = run_layer(H, L, w, b, sc["s_x"], sc["s_out"], 0, False, x, H.IN_I8, ch.s_in)
    assert got.shape == (1, 128, 128, 192)
    assert np.array_equal(got, ref)


# ------------------------------------------------------------------ chains (a5)

def run_chain(H, ch, scales):
    from paper_2608_01653_gb300.chain import Chain
    params = C.chain_params(ch)
    plan = C.plan_chain(ch)
    x = C.chain_input(ch)
    kind = H.IN_F16 if ch.input_kind == "f16" else H.IN_I8
    chain = Chain(ch.layers, params, scales, plan, ch.out_f32)
    outs = chain.forward(dev(x), kind, ch.s_in)
    H.sync_status()
    preps = O.prepare_chain(ch.layers, params, scales, ch.out_f32)
    refs = O.chain_forward(ch.layers, preps, x, ch.input_kind, ch.s_in)
    return [host(o) for o in outs], refs


def test_cfg2_analysis_chain_bit_exact(H):
    ch = C.CONFIGS["cfg2"].chains[0]
    outs, refs = run_chain(H, ch, CALIB["cfg2"][ch.name])
    for i, (g, r) in enumerate(zip(outs, refs)):
        assert np.array_equal(g, r), f"layer {ch.layers[i].name} differs"


@pytest.mark.parametrize("chain_idx", range(9))
def test_cfg3_entropy_chains_bit_exact(H, chain_idx):
    ch = C.CONFIGS["cfg3"].chains[chain_idx]
    outs, refs = run_chain(H, ch, CALIB["cfg3"][ch.name])
    for i, (g, r) in enumerate(zip(outs, refs)):
        assert np.array_equal(g, r), f"{ch.name}/{ch.layers[i].name} differs"
