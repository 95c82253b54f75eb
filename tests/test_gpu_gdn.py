"""GPU parity of the GDN / IGDN transition (Sec. general nonlinearities;
Eqs. supp_general_preactivation, supp_general_activation,
supp_general_input_transition; phi_int of reading R21) through the C ABI,
bit-exact against the oracle: the normalization pool D = B + G z^2 on the
tensor cores, the rounding of R |z| / sqrt(D) (IGDN: R |z| sqrt(D)) decided
by exact comparisons, and the next layer's input transition."""
import numpy as np
import pytest

from oracle import hatq_oracle as O
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


def _params(c, seed, gamma_scale=0.01):
    rng = np.random.default_rng(seed)
    return 0.5 + rng.random(c), np.abs(rng.standard_normal((c, c))) * gamma_scale


def _oracle(z, beta, gamma, s_z, s_u, inverse, s_y, hb_next):
    g = O.gdn_params(beta, gamma, s_z, s_u, inverse)
    g_in = np.sqrt(hb_next) if hb_next else 1.0
    M, n = O.fixed_point([float(np.float32(s_u)) / (g_in * float(np.float32(s_y)))], [127], hb_next if hb_next else 1)
    p = O.Prepared(M_in=int(M[0]), n_in=n, hb_next=hb_next)
    u = O.gdn_int(z, g)
    return O.input_transition(u, p), u


def _codes(shape, seed):
    """Preactivation codes shaped like a conv output: Gaussian, a few
    saturated, whole zero pixels and one pixel of -127."""
    rng = np.random.default_rng(seed)
    z = np.clip(np.rint(rng.normal(0.0, 45.0, shape)), -127, 127).astype(np.int8)
    flat = z.reshape(-1, shape[-1])
    flat[0] = 0
    flat[1] = -127
    flat[2, ::3] = 127
    return z


CASES = [
    # (n, h, w), c, inverse, hb_next
    ((1, 3, 5), 64, False, 0),                        # one partial tile
    ((2, 37, 53), 192, False, 64),                    # 31 tiles, ragged tail
    ((1, 16, 24), 128, True, 32),                     # three full tiles
    ((1, 40, 41), 256, False, 16),                    # one z buffer per CTA
    ((3, 11, 13), 192, True, 0),
    ((1, 7, 9), 64, True, 1),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"{'igdn' if c[2] else 'gdn'}_c{c[1]}_{c[0][0]}x{c[0][1]}x{c[0][2]}")
def test_gdn_transition_bit_exact(H, case):
    (n, h, w), c, inverse, hb_next = case
    beta, gamma = _params(c, c + n)
    z = _codes((n, h, w, c), seed=c * 7 + h)
    s_z, s_y = 0.04, 0.05
    # activation scale from the fp64 model: its max-abs maps to code 135, so the largest codes saturate
    s_u = float(np.float32(np.abs(O.gdn(s_z * z.astype(np.float64), beta, gamma, inverse)).max() / 135.0))
    ref, u = _oracle(z, beta, gamma, s_z, s_u, inverse, s_y, hb_next)
    G = H.prepare_gdn(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next)
    y = H.gdn(dev(z), G)
    H.sync_status()
    got = y.cpu().numpy()
    assert np.array_equal(got, ref)
    assert len(np.unique(u)) > 40 and (np.abs(u) == 127).any()


def test_gdn_gamma_zero_and_all_saturated(H):
    """gamma = 0 (the pool is B alone) and an activation scale so small that
    every nonzero code saturates."""
    c = 128
    beta = np.linspace(0.5, 2.0, c)
    z = _codes((1, 9, 15, c), seed=3)
    for gamma, s_u in ((np.zeros((c, c)), 0.02), (_params(c, 4)[1], 1e-5)):
        ref, u = _oracle(z, beta, gamma, 0.05, s_u, False, 0.04, 64)
        G = H.prepare_gdn(c, beta, gamma, 0.05, s_u, False, 0.04, 64)
        y = H.gdn(dev(z), G)
        H.sync_status()
        assert np.array_equal(y.cpu().numpy(), ref)
    assert np.all(np.abs(u[z != 0]) == 127)


@pytest.mark.parametrize("inverse", [False, True])
def test_conv_then_gdn_matches_oracle_layer(H, inverse):
    """A DH layer (3x3, 192 -> 192) emitting the preactivation z, then the
    transition: equal to the oracle's layer with act gdn / igdn
    (epilogue_general_vector on the oracle's own convolution)."""
    c = 192
    x = I.activations_i8((2, 13, 17, c), seed=21, s_in=0.05)
    w, b = I.weights(c, 3, 3, c, seed=22), I.bias(c, seed=23)
    beta, gamma = _params(c, 24)
    s_x = 0.11
    y_real = O.conv_real(x.astype(np.float64) * 0.05, w, b, 1, 1)
    s_z = float(np.float32(O.symmetric_scale(y_real)))
    u_real = O.gdn(y_real, beta, gamma, inverse)
    s_u = float(np.float32(O.symmetric_scale(u_real)))
    s_y = 0.03
    act = "igdn" if inverse else "gdn"
    p = O.prepare_layer(w, b, "DH", 64, 0, s_x, s_y, act, 64, False, 1, 1, s_z=s_z, s_u=s_u,
                        gdn_beta=beta, gdn_gamma=gamma)
    op = O.quantize_act_i8(x, 64, 0.05, s_x)
    ref = O.epilogue_general_vector(O.conv_codes(op, p.w_int, 1, 1), p)
    L = H.prepare_weights(H.make_desc(c, c, 3, 1, 1, "DH", hb_in=64), w, b, s_x, s_z, "none", 0, False)
    G = H.prepare_gdn(c, beta, gamma, s_z, s_u, inverse, s_y, 64)
    zt = H.conv2d_i8(dev(op), L)
    y = H.gdn(zt, G)
    H.sync_status()
    assert np.array_equal(zt.cpu().numpy(), O.preactivation(O.conv_codes(op, p.w_int, 1, 1), p))
    assert np.array_equal(y.cpu().numpy(), ref)


def test_gdn_binding_rejects_mismatched_tensors(H):
    import torch
    beta, gamma = _params(64, 1)
    G = H.prepare_gdn(64, beta, gamma, 0.05, 0.02, False, 0.05)
    with pytest.raises(ValueError):
        H.gdn(torch.zeros((1, 4, 4, 128), dtype=torch.int8, device="cuda"), G)
    with pytest.raises(ValueError):
        H.gdn(torch.zeros((1, 4, 4, 64), dtype=torch.float16, device="cuda"), G)
    assert H.gdn(torch.zeros((0, 4, 4, 64), dtype=torch.int8, device="cuda"), G).numel() == 0
