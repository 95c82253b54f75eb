"""GPU parity of the decoder-side operators (synthesis transforms), through
the C ABI, bit-exact against the oracle: transposed convolutions as one
stride-1 sub-convolution per output parity class with the output remap in
the copy-out, and the sub-pixel (depth-to-space) rearrangement in the
copy-out. Both are linear operators Y = X W^T (Eq. linear_operator), so the
DH / WH transforms and the integer transition of the analysis layers apply
unchanged (oracle: conv_transpose_layer, depth_to_space)."""
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


def _operand(L, x, s_in):
    """The layer's INT8 operand and its scale (DH: quantized in the input basis)."""
    if L.form == "WH":
        return x, s_in
    y = O.transform_real(x.astype(np.float64) * float(np.float32(s_in)), L.hb_in)
    s_x = float(np.float32(O.symmetric_scale(y)))
    return O.quantize_act_i8(x, L.hb_in, s_in, s_x), s_x


TRANSPOSED = [
    # name, layer (stride / pad of the transposed conv), input (n, h, w), output padding, next block
    ("wh5x5s2_p2_q1", C.layer("t", 192, 192, 5, 2, 2, "WH", "relu", hb_out=64), (2, 9, 14), 1, 64),
    ("dh5x5s2_p2_q1", C.layer("t", 192, 128, 5, 2, 2, "DH", "relu", hb_in=64), (1, 11, 7), 1, 0),
    ("dh4x4s2_p1_q0", C.layer("t", 128, 64, 4, 2, 1, "DH", "none", hb_in=128), (1, 10, 13), 0, 0),
    ("wh3x3s2_p1_q1_next128", C.layer("t", 64, 128, 3, 2, 1, "WH", "relu", hb_out=128), (1, 8, 9), 1, 128),
    ("dh3x3s2_p2_negative_offset", C.layer("t", 64, 64, 3, 2, 2, "DH", "none", hb_in=64), (1, 9, 8), 1, 0),
    ("wh5x5s2_c3_gather", C.layer("t", 3, 64, 5, 2, 2, "WH", "relu", hb_out=32), (1, 12, 15), 1, 0),
    ("dh3x3s1_p1", C.layer("t", 64, 96, 3, 1, 1, "DH", "relu", hb_in=32), (2, 6, 7), 0, 32),
    ("dh5x5s2_c96_pieces", C.layer("t", 96, 64, 5, 2, 2, "DH", "relu", hb_in=32), (1, 8, 9), 1, 0),
]


@pytest.mark.parametrize("case", TRANSPOSED, ids=lambda c: c[0])
@pytest.mark.parametrize("out_f32", [False, True], ids=["int8", "f32"])
def test_transposed_layer_bit_exact(H, case, out_f32):
    name, L, (n, h, w), q, hb_next = case
    if out_f32:
        hb_next = 0
    x = I.activations_i8((n, h, w, L.c_in), seed=len(name) + n, s_in=0.05)
    wts, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=81), I.bias(L.c_out, seed=82)
    op, s_x = _operand(L, x, 0.05)
    y_real = O.conv_transpose_real(x.astype(np.float64) * 0.05, wts, b, L.stride, L.pad, q)
    y_real = np.maximum(y_real, 0) if L.act == "relu" else y_real
    s_y = float(np.float32(O.symmetric_scale(O.transform_real(y_real, hb_next) if hb_next else y_real)))
    T = H.prepare_weights_transposed(H.desc_from_spec(L), q, wts, b, s_x, s_y, L.act, hb_next, out_f32)
    y = H.conv_transpose2d_i8(dev(op), T)
    H.sync_status()
    p = O.prepare_layer(wts, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, out_f32, L.stride, L.pad)
    ref = O.conv_transpose_layer(op, p, q)
    got = y.cpu().numpy()
    assert got.shape == ref.shape
    if out_f32:
        r = np.asarray(ref, np.float64)
        assert np.linalg.norm(got - r) <= 1e-5 * np.linalg.norm(r)
    else:
        assert np.array_equal(got, ref)
        assert np.mean(np.abs(ref.astype(int)) == 127) < 0.2


SUBPIXEL = [
    ("dh3x3_r2", C.layer("s", 64, 256, 3, 1, 1, "DH", "relu", hb_in=64), (2, 9, 11), 2, 0),
    ("wh3x3_r2", C.layer("s", 192, 768, 3, 1, 1, "WH", "relu", hb_out=64), (1, 7, 10), 2, 0),
    ("dh5x5s2_r2", C.layer("s", 64, 128, 5, 2, 2, "DH", "relu", hb_in=64), (1, 13, 10), 2, 0),
]


@pytest.mark.parametrize("case", SUBPIXEL, ids=lambda c: c[0])
def test_subpixel_layer_bit_exact(H, case):
    """Convolution to C r^2 channels, then channel c r^2 + i r + j of pixel
    (oy, ox) to channel c of pixel (oy r + i, ox r + j)."""
    name, L, (n, h, w), r, hb_next = case
    x = I.activations_i8((n, h, w, L.c_in), seed=len(name), s_in=0.05)
    wts, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=83), I.bias(L.c_out, seed=84)
    op, s_x = _operand(L, x, 0.05)
    y_real = np.maximum(O.conv_real(x.astype(np.float64) * 0.05, wts, b, L.stride, L.pad), 0)
    s_y = float(np.float32(O.symmetric_scale(O.transform_real(y_real, hb_next) if hb_next else y_real)))
    P = H.prepare_weights(H.desc_from_spec(L), wts, b, s_x, s_y, L.act, hb_next, False)
    y = H.conv2d_i8_subpixel(dev(op), P, r)
    H.sync_status()
    p = O.prepare_layer(wts, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, False, L.stride, L.pad)
    ref = O.depth_to_space(O.conv_layer(op, p), r)
    assert np.array_equal(y.cpu().numpy(), ref)


def test_subpixel_rejects_what_it_does_not_cover(H):
    L = C.layer("s", 64, 96, 3, 1, 1, "DH", "none", hb_in=64)
    P = H.prepare_weights(H.desc_from_spec(L), I.weights(96, 3, 3, 64, 1), None, 0.1, 0.1)
    x = dev(I.uniform_codes((1, 4, 4, 64), seed=1))
    with pytest.raises(H.HatqError) as e:            # 96 channels: 24 per sub-pixel, not whole 16-groups
        H.conv2d_i8_subpixel(x, P, 2)
    assert e.value.status == H.ERR_UNSUPPORTED
    L = C.layer("s", 64, 256, 3, 1, 1, "DH", "relu", hb_in=64)
    P = H.prepare_weights(H.desc_from_spec(L), I.weights(256, 3, 3, 64, 2), None, 0.1, 0.1, "relu", 64)
    with pytest.raises(H.HatqError) as e:            # a next-layer transform would mix sub-pixels
        H.conv2d_i8_subpixel(x, P, 2)
    assert e.value.status == H.ERR_UNSUPPORTED
