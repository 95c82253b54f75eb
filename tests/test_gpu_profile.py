"""GPU parity of the range-expansion profiling pass (Eq. hadamard_sensitivity)
and the DH/WH selection it drives (Eq. layerwise_hadamard_selection): the
per-image maxima and indicators of hatq_profile_range must equal the oracle's
exactly, on ragged shapes, every block size, many images, and the degenerate
images the statistic has (constant, spike, exact tie, all zero)."""
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


def _check(H, x, hb):
    import torch
    maxima, expands = H.profile_range(torch.from_numpy(np.ascontiguousarray(x)).cuda(), hb)
    H.sync_status()
    mx, mh, ind = O.range_expansion_codes(x, hb)
    got = maxima.cpu().numpy()
    assert np.array_equal(got[:, 0], mx) and np.array_equal(got[:, 1], mh)
    assert np.array_equal(expands.cpu().numpy(), ind)
    p = O.expansion_probability(ind)
    assert H.select_form(expands) == (O.select_form(p), p)          # Eq. layerwise_hadamard_selection, C ABI
    return ind


@pytest.mark.parametrize("shape,hb", [((3, 7, 9, 192), 64), ((2, 5, 3, 256), 256), ((4, 4, 4, 128), 128),
                                      ((5, 3, 5, 32), 32), ((2, 6, 7, 16), 16), ((3, 9, 1, 64), 2),
                                      ((1, 3, 3, 64), 8), ((2, 1, 1, 48), 16), ((2, 33, 17, 320), 64),
                                      ((1, 1, 1, 16), 4)])
def test_profile_bit_exact(H, shape, hb):
    rng = np.random.default_rng(sum(shape) + hb)
    x = I.activations_i8(shape, seed=int(rng.integers(1 << 30)), s_in=0.05)
    x[::2] = np.maximum(x[::2], 0)            # ReLU-like images: nonzero channel means
    _check(H, x, hb)


def test_profile_degenerate_images(H):
    x = np.zeros((5, 2, 3, 64), np.int8)
    x[0] = -9                                   # constant: expands by sqrt(hb)
    x[1, 1, 2, 7] = 127                         # one spike: shrinks
    x[2, 0, 0, :4] = (1, 1, 0, 0)               # exact tie at hb = 4: not an expansion
    x[3] = np.tile(np.array([127, -127], np.int8), 32)   # a Hadamard row: accumulates like a mean
    ind = _check(H, x, 4)                       # image 4 stays all zero
    assert ind.tolist() == [1, 0, 0, 1, 0]
    _check(H, x, 64)


def test_profile_many_images_and_selection(H):
    """M = 70 images, a mix that puts p_l on both sides of tau_sel = 0.8."""
    rng = np.random.default_rng(11)
    x = rng.integers(-3, 4, size=(70, 6, 10, 64)).astype(np.int8)
    x[:, :, :, 9] = 110                         # an outlier channel: the transform spreads it
    shifted = np.clip(np.maximum(x[:50].astype(np.int16), 0) + 40, -127, 127)
    x[:50] = shifted.astype(np.int8)           # 50 nonnegative images: coherent mean
    ind = _check(H, x, 64)
    assert 0 < ind.sum() < 70


def test_profile_config4_layer_input_sample(H):
    """The ga2 input shape of the benchmark workload at one image and a crop
    of 270x480, checked against the oracle."""
    x = I.activations_i8((1, 270, 480, 192), seed=5, s_in=0.05)
    _check(H, x, 64)


def test_profile_empty_batch_and_bad_arguments(H):
    import torch
    m, e = H.profile_range(torch.zeros((0, 4, 4, 64), dtype=torch.int8, device="cuda"), 64)
    assert m.shape == (0, 2) and e.shape == (0,)
    for hb in (3, 512):
        with pytest.raises(H.HatqError):
            H.profile_range(torch.zeros((1, 4, 4, 64), dtype=torch.int8, device="cuda"), hb)
    with pytest.raises(H.HatqError):
        H.profile_range(torch.zeros((1, 4, 4, 40), dtype=torch.int8, device="cuda"), 8)
