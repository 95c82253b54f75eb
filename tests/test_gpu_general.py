"""GPU parity of the transition through non-homogeneous activations (SiLU,
GELU; Sec. general nonlinearities): preactivation codes, integer table and
input-side rescale with the fused next transform, bit-exact against the
oracle across forms, fused and unfused transitions, reductions that drain in
several exact chunks, and the small-channel gather."""
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


CASES = [
    # name, layer, input (n, h, w), hb_next
    ("dh3x3_silu", C.layer("a", 64, 64, 3, 1, 1, "DH", "silu", hb_in=64), (2, 9, 13), 0),
    ("wh3x3_gelu_next64", C.layer("a", 64, 128, 3, 1, 1, "WH", "gelu", hb_out=64), (1, 11, 17), 64),
    ("dh5x5s2_gelu_next32_drain", C.layer("a", 192, 192, 5, 2, 2, "DH", "gelu", hb_in=64), (1, 19, 37), 32),
    ("wh5x5s2_c3_silu_gather", C.layer("a", 3, 64, 5, 2, 2, "WH", "silu", hb_out=32), (2, 30, 41), 64),
    ("dh1x1_silu_ragged", C.layer("a", 128, 224, 1, 1, 0, "DH", "silu", hb_in=128), (3, 5, 7), 32),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_general_layer_bit_exact(H, case):
    import torch
    name, L, (n, h, w), hb_next = case
    wts = I.weights(L.c_out, L.k, L.k, L.c_in, seed=41)
    b = I.bias(L.c_out, seed=42)
    x_real = np.maximum(I.activations((n, h, w, L.c_in), seed=43).astype(np.float64), 0)
    y = O.conv_real(x_real, wts, b, L.stride, L.pad)
    u = np.vectorize(lambda v: O.phi(L.act, v))(y)
    s_x = O.symmetric_scale(O.transform_real(x_real, L.hb_in)) if L.form == "DH" else O.symmetric_scale(x_real)
    tgt = O.transform_real(u, hb_next) if hb_next else u
    s_x, s_z, s_u, s_y = (float(np.float32(v)) for v in
                          (s_x, O.symmetric_scale(y), O.symmetric_scale(u), O.symmetric_scale(tgt)))
    op = O.quantize_act_f16(x_real.astype(np.float16), L.hb_in if L.form == "DH" else 1, s_x)
    P = H.prepare_weights(H.desc_from_spec(L), wts, b, s_x, s_y, L.act, hb_next, s_z=s_z, s_u=s_u)
    got = H.conv2d_i8(torch.from_numpy(op).cuda(), P)
    H.sync_status()
    ref_p = O.prepare_layer(wts, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, False, L.stride, L.pad,
                            s_z=s_z, s_u=s_u)
    ref = O.conv_layer(op, ref_p)
    assert np.array_equal(got.cpu().numpy(), ref)
    assert np.mean(np.abs(ref.astype(int)) == 127) < 0.2


def test_general_layer_rejects_float_output(H):
    L = C.layer("a", 64, 64, 3, 1, 1, "DH", "silu", hb_in=64)
    with pytest.raises(ValueError):
        H.prepare_weights(H.desc_from_spec(L), np.zeros((64, 3, 3, 64), np.float32), None, 0.1, 0.1, "silu", 0,
                          out_f32=True, s_z=0.1, s_u=0.1)
