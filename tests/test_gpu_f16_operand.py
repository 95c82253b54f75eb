"""GPU parity of the fp16 storage of INT8 codes (hatq_set_operand_format):
a layer whose operand arrives as fp16 values (the tensor cores read the TMA
tile in shared memory, no per-tile conversion) and a layer that writes its
codes as fp16 compute the same codes as the INT8 path, bit for bit against
the oracle; a chain with fp16 operands equals the INT8 chain."""
import zlib

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


CASES = [
    # name, layer, input (n, h, w), hb_next
    ("dh3x3_drain_next64", C.layer("a", 192, 192, 3, 1, 1, "DH", "relu", hb_in=64), (2, 13, 37), 64),
    ("dh5x5s2_ragged", C.layer("a", 192, 192, 5, 2, 2, "DH", "none", hb_in=64), (3, 19, 45), 0),
    ("wh3x3_c640_128_next128", C.layer("a", 320, 640, 3, 1, 1, "WH", "relu", hb_out=128), (1, 7, 10), 128),
    ("wh3x3_256_128_next128", C.layer("a", 256, 128, 3, 1, 1, "WH", "relu", hb_out=128), (2, 11, 21), 128),
    ("dh3x3_c64_box", C.layer("a", 64, 224, 3, 1, 1, "DH", "relu", hb_in=32), (2, 9, 17), 0),
    ("dh1x1_c640_n5", C.layer("a", 640, 640, 1, 1, 0, "DH", "none", hb_in=128), (1, 9, 23), 0),
]


def _layer(case):
    name, L, (n, h, w), hb_next = case
    seed = zlib.crc32(name.encode()) % 1000
    x = I.activations_i8((n, h, w, L.c_in), seed=seed, s_in=0.05)
    wts, b = I.weights(L.c_out, L.k, L.k, L.c_in, seed=seed + 1), I.bias(L.c_out, seed=seed + 2)
    if L.form == "WH":
        s_x, op = 0.05, x
    else:
        y = O.transform_real(x.astype(np.float64) * float(np.float32(0.05)), L.hb_in)
        s_x = float(np.float32(O.symmetric_scale(y)))
        op = O.quantize_act_i8(x, L.hb_in, 0.05, s_x)
    s_y = 0.07
    p = O.prepare_layer(wts, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, hb_next, False, L.stride, L.pad)
    return L, wts, b, s_x, s_y, hb_next, op, O.conv_layer(op, p)


@pytest.mark.parametrize("out_f16", [False, True], ids=["i8_out", "f16_out"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_f16_operand_layer_bit_exact(H, case, out_f16):
    import torch
    L, wts, b, s_x, s_y, hb_next, op, ref = _layer(case)
    P = H.prepare_weights(H.desc_from_spec(L), wts, b, s_x, s_y, L.act, hb_next, False)
    H.set_operand_format(P, True, out_f16)
    y = H.conv2d_i8(dev(op).to(torch.float16), P)
    H.sync_status()
    assert y.dtype == (torch.float16 if out_f16 else torch.int8)
    got = y.cpu().numpy()
    assert np.array_equal(got.astype(np.int64), ref.astype(np.int64))
    assert len(np.unique(ref)) > 16


def test_f16_output_of_an_int8_layer(H):
    import torch
    L, wts, b, s_x, s_y, hb_next, op, ref = _layer(CASES[0])
    P = H.prepare_weights(H.desc_from_spec(L), wts, b, s_x, s_y, L.act, hb_next, False)
    H.set_operand_format(P, False, True)
    y = H.conv2d_i8(dev(op), P)
    H.sync_status()
    assert y.dtype == torch.float16 and np.array_equal(y.cpu().numpy().astype(np.int64), ref.astype(np.int64))


def test_f16_operand_rejections(H):
    import torch
    L = C.layer("a", 3, 64, 3, 1, 1, "WH", "relu", hb_out=64)
    P = H.prepare_weights(H.desc_from_spec(L), I.weights(64, 3, 3, 3, 1), None, 0.05, 0.05, "relu", 0, False)
    with pytest.raises(H.HatqError) as e:                    # small-channel (gather) layer
        H.set_operand_format(P, True, False)
    assert e.value.status == H.ERR_UNSUPPORTED
    for c_in in (32, 224):                                   # taps packed at 32-channel granularity
        L = C.layer("a", c_in, 64, 3, 1, 1, "DH", "none", hb_in=32)
        P = H.prepare_weights(H.desc_from_spec(L), I.weights(64, 3, 3, c_in, 1), None, 0.05, 0.05, "none", 0, False)
        with pytest.raises(H.HatqError) as e:
            H.set_operand_format(P, True, False)
        assert e.value.status == H.ERR_UNSUPPORTED
        H.set_operand_format(P, False, True)                 # the fp16 output format is still open
    L = CASES[0][1]
    P = H.prepare_weights(H.desc_from_spec(L), I.weights(192, 3, 3, 192, 2), None, 0.1, 0.1, "relu", 64, False)
    H.set_operand_format(P, True, False)
    x = torch.zeros((1, 8, 8, 192), dtype=torch.int8, device="cuda")
    with pytest.raises(ValueError):                          # the operand must be fp16 now
        H.conv2d_i8(x, P)
    with pytest.raises(H.HatqError) as e:                    # it is the operand, not codes to transform
        H.layer(x.to(torch.float16), H.IN_F16, 0.05, P)
    assert e.value.status == H.ERR_UNSUPPORTED
    assert H.layer_launches(H.IN_I8, 0.05, P) == -1


def test_chain_with_f16_operands_equals_int8_chain(H):
    """The config-3 hyperprior chain (320 -> 640 -> 640 -> 640, the 640-wide
    layers taking fp16 operands) gives the same codes as the INT8 chain."""
    import json
    import os
    import torch
    from paper_2608_01653_gb300.chain import Chain
    calib = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "calibration.json")))["configs"]
    ch = [c for c in C.CONFIGS["cfg3"].chains if c.name == "hyper"][0]
    params = C.chain_params(ch)
    sc = calib["cfg3"][ch.name]
    x = torch.from_numpy(C.chain_input(ch)).cuda()
    base = Chain(ch.layers, params, sc, C.plan_chain(ch), ch.out_f32).forward(x, H.IN_I8, ch.s_in)
    f16 = Chain(ch.layers, params, sc, C.plan_chain(ch), ch.out_f32, f16_operands=(1, 2)).forward(x, H.IN_I8, ch.s_in)
    H.sync_status()
    assert f16[0].dtype == torch.float16 and f16[1].dtype == torch.float16
    for a, b in zip(base, f16):
        assert np.array_equal(a.cpu().numpy().astype(np.int64), b.cpu().numpy().astype(np.int64))
