"""hatq_layer_noalloc, the entry point for callers that cannot allocate device
memory (host callbacks, plugins whose host engine owns every allocation,
allocator-less embeddings): it stages the layer's INT8 operand in the
library's fixed device array instead of a caller scratch buffer.

Checked through the C ABI against hatq_layer (which takes caller scratch) on
two calls in a row with different inputs, so contents left in the shared
array by one call cannot leak into the next. Collected last on purpose."""
import numpy as np
import pytest

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


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def test_noalloc_matches_layer_int8_path_two_calls(H):
    desc = H.make_desc(192, 192, 5, 2, 2, "DH", hb_in=64)
    w, b = I.weights(192, 5, 5, 192, 21), I.bias(192, 22)
    L = H.prepare_weights(desc, w, b, 0.11, 0.05, "relu", 64, False)
    for seed in (1, 2):                               # two calls in a row, different inputs
        x = _dev(I.activations_i8((2, 40, 56, 192), seed=seed, s_in=0.05))
        ref = H.layer(x, H.IN_I8, 0.05, L)
        got = H.layer_noalloc(x, H.IN_I8, 0.05, L)
        H.sync_status()
        assert np.array_equal(got.cpu().numpy(), ref.cpu().numpy())


def test_noalloc_matches_layer_fp16_entry_two_calls(H):
    desc = H.make_desc(128, 128, 1, 1, 0, "DH", hb_in=128)
    w, b = I.weights(128, 1, 1, 128, 23), I.bias(128, 24)
    L = H.prepare_weights(desc, w, b, 0.7, 1.0, "none", 0, True)
    for seed in (3, 4):
        x = _dev(I.activations_f16((1, 16, 16, 128), seed=seed))
        ref = H.layer(x, H.IN_F16, 1.0, L).cpu().numpy().astype(np.float64)
        got = H.layer_noalloc(x, H.IN_F16, 1.0, L).cpu().numpy().astype(np.float64)
        H.sync_status()
        assert np.linalg.norm(got - ref) <= 1e-3 * np.linalg.norm(ref)


def test_noalloc_operand_input_and_size_limit(H):
    import torch
    desc = H.make_desc(192, 192, 5, 2, 2, "DH", hb_in=64)
    L = H.prepare_weights(desc, I.weights(192, 5, 5, 192, 25), None, 0.11, 0.05)
    x = _dev(I.uniform_codes((1, 20, 24, 192), seed=5))
    got = H.layer_noalloc(x, H.IN_OPERAND, 0.0, L)   # already the operand: nothing staged
    ref = H.layer(x, H.IN_OPERAND, 0.0, L)
    H.sync_status()
    assert np.array_equal(got.cpu().numpy(), ref.cpu().numpy())
    big = torch.zeros((1, 448, 448, 192), dtype=torch.int8, device="cuda")   # 38.5 MB > 32 MiB
    assert big.numel() > H.NOALLOC_MAX_BYTES
    with pytest.raises(H.HatqError) as e:
        H.layer_noalloc(big, H.IN_I8, 0.05, L)
    assert e.value.status == H.ERR_INVALID_ARG and "HATQ_NOALLOC_MAX_BYTES" in H.last_error()
