"""GPU parity of the paper's single Hadamard order m(C) (Supp. Hadamard
construction; Eqs. supp_hadamard_order, supp_padded_transforms,
supp_padded_dh): the activation-side transform as a bias-free 1x1
convolution on the tensor cores (supplementary, deployment realization) and
DH layers whose weights carry the order-m transform, through the C ABI,
bit-exact against the oracle. Orders: Paley-I 192 and 224, the Kronecker
products 96 and 320, and 190 channels zero-padded to 192."""
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


def _scale_of_order(x_i8, s_in, m):
    y = O.transform_order_real(np.asarray(x_i8, np.float64) * float(np.float32(s_in)), m)
    return float(np.float32(O.symmetric_scale(y)))


@pytest.mark.parametrize("shape", [(2, 13, 17, 192), (1, 9, 31, 190), (1, 7, 9, 224), (3, 5, 6, 320),
                                   (1, 11, 5, 96)])
def test_order_transform_layer_bit_exact(H, shape):
    c = shape[-1]
    m = O.hadamard_order(c)
    x = I.activations_i8(shape, seed=c + shape[1], s_in=0.05)
    x[0, 0, 0, :] = 127                              # the coherent worst case |y| = 127 c
    s_out = _scale_of_order(x, 0.05, m)
    T = H.prepare_order_transform(c, 0.05, s_out)
    y = H.layer(dev(x), H.IN_I8, 0.05, T)
    H.sync_status()
    ref = O.quantize_act_order_i8(x, m, 0.05, s_out)
    assert y.shape[-1] == m
    assert np.array_equal(y.cpu().numpy(), ref)
    assert np.abs(ref.astype(int)).max() == 127


ORDER_LAYERS = [
    ("dh5x5s2_c192", C.layer("a", 192, 192, 5, 2, 2, "DH", "relu", hb_in=64), (2, 19, 27), 0),
    ("dh3x3_c190_pad", C.layer("a", 190, 64, 3, 1, 1, "DH", "none", hb_in=2), (1, 14, 11), 0),
    ("dh3x3_c320_kron_next128", C.layer("a", 320, 640, 3, 1, 1, "DH", "relu", hb_in=64), (1, 6, 9), 128),
    ("dh3x3_c224_next32", C.layer("a", 224, 128, 3, 1, 1, "DH", "relu", hb_in=32), (1, 10, 13), 32),
    ("dh1x1_c96_kron", C.layer("a", 96, 128, 1, 1, 0, "DH", "none", hb_in=32), (2, 8, 8), 0),
]


@pytest.mark.parametrize("case", ORDER_LAYERS, ids=lambda c: c[0])
def test_order_layer_bit_exact(H, case):
    """Transform layer then the order-m DH layer, both on the GPU, against
    the oracle's order quantizer and the layer prepared with order_in = m."""
    name, L, (n, h, w), hb_next = case
    m = O.hadamard_order(L.c_in)
    x = I.activations_i8((n, h, w, L.c_in), seed=len(name), s_in=0.05)
    wts, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=71), I.bias(L.c_out, seed=72)
    s_x = _scale_of_order(x, 0.05, m)
    y_real = O.conv_real(x.astype(np.float64) * 0.05, wts, b, L.stride, L.pad)
    y_real = np.maximum(y_real, 0) if L.act == "relu" else y_real
    s_y = float(np.float32(O.symmetric_scale(O.transform_real(y_real, hb_next) if hb_next else y_real)))
    T = H.prepare_order_transform(L.c_in, 0.05, s_x)
    P = H.prepare_weights_order(H.make_desc(L.c_in, L.c_out, L.k, L.stride, L.pad, "DH"), wts, b, s_x, s_y, L.act,
                                hb_next)
    op = H.layer(dev(x), H.IN_I8, 0.05, T)
    y = H.layer(op, H.IN_OPERAND, s_x, P)
    H.sync_status()
    ref_op = O.quantize_act_order_i8(x, m, 0.05, s_x)
    assert np.array_equal(op.cpu().numpy(), ref_op)
    pr = O.prepare_layer(wts, b, "DH", 0, 0, s_x, s_y, L.act, hb_next, False, L.stride, L.pad, order_in=m)
    ref = O.conv_layer(ref_op, pr)
    assert np.array_equal(y.cpu().numpy(), ref)
    assert np.mean(np.abs(ref.astype(int)) == 127) < 0.2


def test_order_layer_rejects_unordered_input(H):
    L = ORDER_LAYERS[0][1]
    P = H.prepare_weights_order(H.make_desc(192, 192, 5, 2, 2, "DH"), I.weights(192, 5, 5, 192, 1), None, 0.1, 0.1)
    x = dev(I.activations_i8((1, 8, 8, 192), seed=1, s_in=0.05))
    with pytest.raises(H.HatqError) as e:
        H.layer(x, H.IN_I8, 0.05, P)
    assert e.value.status == H.ERR_UNSUPPORTED and L.c_in == 192


def test_paper_order_analysis_chain_bit_exact(H):
    """The config-2 analysis chain (768x512 image, 3->192->192->192->320) with
    the paper's orders on the DH side: ga1 (WH, Sylvester 64 on the output
    side) emits original-basis codes; before each DH layer the order-192
    transform layer (Paley-I, q = 191) moves them into that layer's basis, as
    in the supplementary's deployment realization. Every tensor is compared."""
    ch = C.CONFIGS["cfg2"].chains[0]
    params = C.chain_params(ch)
    x = C.chain_input(ch)
    x_real = x.astype(np.float64) * float(np.float32(ch.s_in))
    # static scales from the fp64 model: original-basis outputs, order-basis operands
    reals, cur = [], x_real
    for L, (w, b) in zip(ch.layers, params):
        y = O.conv_real(cur, w, b, L.stride, L.pad)
        cur = np.maximum(y, 0) if L.act == "relu" else y
        reals.append(cur)
    s_out = [float(np.float32(O.symmetric_scale(r))) for r in reals]
    m = O.hadamard_order(192)
    s_op = [float(np.float32(O.symmetric_scale(O.transform_order_real(reals[i - 1], m)))) for i in (1, 2, 3)]

    ga1 = ch.layers[0]
    P1 = H.prepare_weights(H.desc_from_spec(ga1), params[0][0], params[0][1], ch.s_in, s_out[0], "relu", 0)
    y = H.layer(dev(x), H.IN_I8, ch.s_in, P1)
    r1 = O.prepare_layer(params[0][0], params[0][1], "WH", 0, ga1.hb_out, ch.s_in, s_out[0], "relu", 0, False,
                         ga1.stride, ga1.pad)
    ref = O.conv_layer(x, r1)
    H.sync_status()
    assert np.array_equal(y.cpu().numpy(), ref), "ga1"
    for i in (1, 2, 3):
        L = ch.layers[i]
        w, b = params[i]
        T = H.prepare_order_transform(192, s_out[i - 1], s_op[i - 1])
        P = H.prepare_weights_order(H.make_desc(192, L.c_out, L.k, L.stride, L.pad, "DH"), w, b, s_op[i - 1],
                                    s_out[i], L.act, 0)
        op = H.layer(y, H.IN_I8, s_out[i - 1], T)
        y = H.layer(op, H.IN_OPERAND, s_op[i - 1], P)
        H.sync_status()
        ref_op = O.quantize_act_order_i8(ref, m, s_out[i - 1], s_op[i - 1])
        assert np.array_equal(op.cpu().numpy(), ref_op), f"{L.name} operand"
        pr = O.prepare_layer(w, b, "DH", 0, 0, s_op[i - 1], s_out[i], L.act, 0, False, L.stride, L.pad, order_in=m)
        ref = O.conv_layer(ref_op, pr)
        assert np.array_equal(y.cpu().numpy(), ref), L.name
