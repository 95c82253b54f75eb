"""Failure detection on the GPU without a fault: a bounded device wait is made
to expire on purpose (hatq_selftest_wait waits, through the convolution
pipeline's own bounded mbarrier wait, on a barrier nothing arrives at). The
expiry must surface as HATQ_ERR_TIMEOUT from hatq_sync_status, convolutions
enqueued behind it must be skipped rather than run on a poisoned pipeline, and
the library must give correct results again once the status was read."""
import numpy as np
import pytest

from oracle import hatq_oracle as O
from synth import configs as C
from synth import inputs as I

pytestmark = pytest.mark.gpu

LIMIT = 2_000_000          # cycles: about a millisecond


@pytest.fixture(scope="module")
def H():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_01653_gb300 import hatq
    hatq.load()
    hatq.sync_status()
    return hatq


def _layer(H):
    import torch
    L = C.layer("a", 64, 64, 3, 1, 1, "DH", "relu", hb_in=64)
    w = I.weights(64, 3, 3, 64, seed=21)
    b = I.bias(64, seed=22)
    x = I.activations_i8((1, 12, 20, 64), seed=23, s_in=0.05)
    s_x, s_y = 0.02, 0.05
    P = H.prepare_weights(H.desc_from_spec(L), w, b, s_x, s_y, L.act, 0, False)
    ref_p = O.prepare_layer(w, b, L.form, L.hb_in, L.hb_out, s_x, s_y, L.act, 0, False, L.stride, L.pad)
    ref = O.conv_layer(x, ref_p)
    return P, torch.from_numpy(x).cuda(), ref


def test_expired_wait_reports_timeout_then_clears(H):
    H.selftest_wait(LIMIT)
    with pytest.raises(H.HatqError) as e:
        H.sync_status()
    assert e.value.status == H.ERR_TIMEOUT
    assert "bounded wait" in H.last_error()
    H.sync_status()                      # read once: the word is clear again


def test_work_behind_an_expiry_is_skipped_and_the_library_recovers(H):
    import torch
    P, x, ref = _layer(H)
    y = torch.full(P.out_shape(1, 12, 20), 77, dtype=torch.int8, device="cuda")
    H.selftest_wait(LIMIT)
    H.conv2d_i8(x, P, y=y)               # enqueued behind the expiring wait
    with pytest.raises(H.HatqError) as e:
        H.sync_status()
    assert e.value.status == H.ERR_TIMEOUT
    assert bool((y == 77).all()), "a convolution ran although the error word was set"
    H.conv2d_i8(x, P, y=y)
    H.sync_status()
    assert np.array_equal(y.cpu().numpy(), ref)


def test_selftest_rejects_out_of_range_limits(H):
    for bad in (0, 4_000_000_001):
        with pytest.raises(H.HatqError) as e:
            H.selftest_wait(bad)
        assert e.value.status == H.ERR_INVALID_ARG
