"""GPU parity of the dynamic affine activation path (PTQ setting; Eqs.
uniform_q, affine_q; supplementary, affine activation quantization): per
input tensor s and z from its range (zero kept representable), the
convolution on the centred codes x_int - z with zero padding as a centred
zero, and the dequantized output y = phi(H_out(s s_w (.) a) + b_bar).

The integer part is checked exactly: the oracle's convolution takes the
GPU's own centred codes and step, and the GPU output matches it to float32
rounding. The FP16-entry quantizer (an fp32 butterfly against the oracle's
fp64 transform) is held to the FP16-entry tolerance: at most one code step on
at most 0.1 % of codes, and the whole layer to relative L2 error 1e-3."""
import numpy as np
import pytest

from oracle import hatq_oracle as O
from synth import configs as C
from synth import inputs as I

pytestmark = pytest.mark.gpu


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


def rel_l2(got, ref):
    ref = np.asarray(ref, np.float64)
    return float(np.linalg.norm(np.asarray(got, np.float64) - ref) / max(np.linalg.norm(ref), 1e-300))


CASES = [
    ("dh3x3_hb64_relu", C.layer("a", 192, 128, 3, 1, 1, "DH", "relu", hb_in=64), (2, 11, 13), "shifted"),
    ("dh5x5s2_hb64", C.layer("a", 192, 192, 5, 2, 2, "DH", "none", hb_in=64), (1, 21, 30), "signed"),
    ("wh3x3_hb128_relu", C.layer("a", 128, 128, 3, 1, 1, "WH", "relu", hb_out=128), (1, 12, 17), "relu"),
    ("wh1x1_hb64_drain", C.layer("a", 640, 192, 1, 1, 0, "WH", "none", hb_out=64), (1, 9, 7), "signed"),
    ("dh3x3_k2304_drains", C.layer("a", 256, 64, 3, 1, 1, "DH", "relu", hb_in=128), (1, 8, 9), "relu"),
    ("dh3x3_c96_pieces", C.layer("a", 96, 64, 3, 1, 1, "DH", "relu", hb_in=32), (1, 10, 14), "shifted"),
]


def _input(kind, shape, seed):
    x = I.activations(shape, seed=seed).astype(np.float64)
    if kind == "relu":
        x = np.maximum(x, 0)                      # nonnegative: z = 0, the whole grid on one side
    elif kind == "shifted":
        x = x + 2.0                               # off-centre range: z far from 128
    return x.astype(np.float16)


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_affine_layer(H, case):
    name, L, (n, h, w), kind = case
    x = _input(kind, (n, h, w, L.c_in), seed=len(name))
    wts, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=91), I.bias(L.c_out, seed=92)
    hb = L.hb_in if L.form == "DH" else 1
    codes, params = H.quantize_act_affine(dev(x), hb)
    P = H.prepare_weights_affine(H.desc_from_spec(L), wts, b, L.act)
    y = H.conv2d_affine(codes, P, params)
    H.sync_status()
    s_gpu, z_gpu = [float(v) for v in params.cpu().numpy()]
    c_gpu = codes.cpu().numpy().astype(np.int64)
    p = O.prepare_layer(wts, b, L.form, L.hb_in, L.hb_out, 1.0, 1.0, L.act, 0, True, L.stride, L.pad)
    # 1. the quantizer against the oracle's (fp64 transform of the same fp16 input)
    v = O.transform_real(x.astype(np.float64), L.hb_in) if L.form == "DH" else x.astype(np.float64)
    s_ref, z_ref = O.affine_params(v)
    assert abs(s_gpu - s_ref) <= 1e-6 * s_ref and abs(z_gpu - z_ref) <= 1
    c_ref = O.quantize_affine(v, s_ref, z_ref) - z_ref
    d = np.abs(c_gpu - c_ref)
    assert d.max() <= 1 and np.mean(d > 0) <= 1e-3
    assert np.abs(c_gpu).max() <= 255 and (c_gpu + z_gpu).min() >= 0 and (c_gpu + z_gpu).max() <= 255
    # 2. the integer convolution and float epilogue exactly, on the GPU's own codes and step
    got = y.cpu().numpy()
    ref = O.conv_layer_affine_codes(c_gpu, s_gpu, p)
    assert got.shape == ref.shape and rel_l2(got, ref) <= 1e-5
    # 3. end to end against the oracle's path
    ref_e2e, _, _ = O.conv_layer_affine(x.astype(np.float64), p)
    assert rel_l2(got, ref_e2e) <= 1e-3


def test_affine_zero_input_and_wrong_entry(H):
    L = C.layer("a", 64, 64, 3, 1, 1, "DH", "none", hb_in=64)
    codes, params = H.quantize_act_affine(dev(np.zeros((1, 5, 6, 64), np.float16)), 64)
    H.sync_status()
    assert not codes.cpu().numpy().any() and params.cpu().numpy().tolist() == [1.0, 0.0]
    P = H.prepare_weights_affine(H.desc_from_spec(L), I.weights(64, 3, 3, 64, 1), I.bias(64, 2))
    with pytest.raises(H.HatqError):                 # an affine layer is not an INT8-operand layer
        H.conv2d_i8(dev(np.zeros((1, 5, 6, 64), np.int8)), P)
