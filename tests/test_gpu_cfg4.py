"""GPU parity on config 4, the benchmark workload: the LIC analysis chain
(3->192->192->192->320, 5x5 s2) and the entropy-model chains (hyperprior and
8 context slices) at batch 8 on 3840x2160 images (latent 240x135), run
through Chain.forward exactly as the benchmark runs them.

Every layer of every chain is compared with the oracle bit for bit at
sampled output pixels, the oracle taking the GPU's own input of that layer
(so each layer is checked on the tensors the benchmark really produces):
all 8 images, the four image corners, pixels on both sides of every tile
width the library may pick, the last tiles of each image (ragged tails) and
random interior pixels; every output channel of each sampled pixel. Byte
offsets of the largest tensors pass 2^31 (the ga1 output is 3.2 GB), so the
64-bit addressing of the persistent tile loop is exercised. One full image
of the analysis chain is also compared end to end with the oracle's chain."""
import json
import os

import numpy as np
import pytest

from oracle import hatq_oracle as O
from synth import configs as C

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
CALIB = json.load(open(os.path.join(GOLDEN, "calibration.json")))["configs"]
TILE_WIDTHS = (8, 16, 32, 64, 128)


def _scales(ch):
    return CALIB["cfg2" if ch.name == "analysis" else "cfg3"][ch.name]


@pytest.fixture(scope="module")
def run():
    """The whole config-4 step on the GPU; per chain its spec, host input and
    the device outputs of every layer."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_01653_gb300 import hatq as H
    from paper_2608_01653_gb300.chain import Chain
    H.load()
    out = []
    for ch in C.CONFIGS["cfg4"].chains:
        params = C.chain_params(ch)
        chain = Chain(ch.layers, params, _scales(ch), C.plan_chain(ch), ch.out_f32)
        x = C.chain_input(ch)
        outs = chain.forward(torch.from_numpy(x).cuda(), H.IN_I8, ch.s_in)
        out.append((ch, params, x, outs))
    H.sync_status()
    return out


def sample_pixels(n, ho, wo, seed, per_image=160):
    """(b, oy, ox) output pixels: corners, both sides of every tile width,
    the last row and column, the last 128 pixels of each image, random ones."""
    rng = np.random.default_rng(seed)
    pix = []
    for b in range(n):
        pts = {(0, 0), (0, wo - 1), (ho - 1, 0), (ho - 1, wo - 1)}
        for t in TILE_WIDTHS:
            for m in range(1, (wo - 1) // t + 1):
                if rng.random() < 4.0 / max(1, (wo - 1) // t):
                    oy = int(rng.integers(ho))
                    pts.add((oy, m * t - 1))
                    pts.add((oy, m * t))
            for m in range(1, (ho - 1) // t + 1):
                if rng.random() < 2.0 / max(1, (ho - 1) // t):
                    ox = int(rng.integers(wo))
                    pts.add((m * t - 1, ox))
                    pts.add((m * t, ox))
        last = ho * wo - 1 - rng.choice(min(128, ho * wo), size=min(24, ho * wo), replace=False)
        pts.update((int(p // wo), int(p % wo)) for p in last)
        for _ in range(6):
            pts.add((ho - 1, int(rng.integers(wo))))
            pts.add((int(rng.integers(ho)), wo - 1))
        while len(pts) < per_image:
            pts.add((int(rng.integers(ho)), int(rng.integers(wo))))
        pix.extend((b, oy, ox) for oy, ox in sorted(pts))
    return np.array(pix, dtype=np.int64)


def _check_chain(ch, params, x, outs):
    preps = O.prepare_chain(ch.layers, params, _scales(ch), ch.out_f32)
    cur = O.layer_operand(x, "i8", ch.s_in, ch.layers[0].form, ch.layers[0].hb_in, preps[0].s_x)
    for i, (L, p) in enumerate(zip(ch.layers, preps)):
        y = outs[i]
        n, ho, wo, co = y.shape
        pix = sample_pixels(n, ho, wo, seed=1000 + 31 * i + len(ch.name))
        acc = O.conv_codes_at(cur, p.w_int, p.stride, p.pad, pix)
        ref = O.epilogue_int(acc, p)
        got = y.cpu().numpy()
        if got.dtype == np.float16:                       # codes stored as fp16 for an fp16-operand layer
            got = got.astype(np.int8)
        sel = got[pix[:, 0], pix[:, 1], pix[:, 2], :]
        bad = np.argwhere(sel != ref)
        assert bad.size == 0, (f"{ch.name}/{L.name}: {len(bad)} of {ref.size} sampled codes differ, first at pixel "
                               f"{pix[bad[0][0]].tolist()} channel {bad[0][1]}")
        assert len(np.unique(ref)) > 8, f"{ch.name}/{L.name}: degenerate sample"
        cur = got


@pytest.mark.parametrize("idx", range(9), ids=lambda i: C.CONFIGS["cfg4"].chains[i].name)
def test_cfg4_sampled_bit_exact(run, idx):
    ch, params, x, outs = run[idx]
    assert len(outs) == len(ch.layers)
    _check_chain(ch, params, x, outs)


def test_cfg4_offsets_pass_2_31(run):
    ch, _, _, outs = run[0]
    assert ch.name == "analysis" and outs[0].numel() > 2 ** 31


def test_cfg4_analysis_image0_end_to_end(run):
    """Image 0 of the batch through the oracle's whole analysis chain (no
    GPU data in the oracle's path) equals the GPU's outputs of every layer."""
    ch, params, x, outs = run[0]
    preps = O.prepare_chain(ch.layers, params, _scales(ch), ch.out_f32)
    refs = O.chain_forward(ch.layers, preps, x[:1], ch.input_kind, ch.s_in)
    for i, (g, r) in enumerate(zip(outs, refs)):
        assert np.array_equal(g[:1].cpu().numpy().astype(np.int64), r.astype(np.int64)), \
            f"layer {ch.layers[i].name} differs on image 0"
