"""Writes tests/golden/calibration.json: the static per-layer activation
scales of every chain in configs 0-3, calibrated on the real-valued (fp64)
model by the CPU oracle only (frozen tensor-wise scales, as in the paper's QAT
deployment). Config 4 reuses the config-2/3 scales of the same chains.

Run:  python tests/golden/make_calibration.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import hatq_oracle as O  # noqa: E402
from synth import configs as C  # noqa: E402


def real_input(chain, x):
    if chain.input_kind == "f16":
        return x.astype(np.float64)
    return x.astype(np.float64) * float(np.float32(chain.s_in))


def main():
    out = {"note": "per chain, per layer: s_x = scale of the INT8 operand the layer consumes; "
                   "s_out = scale of the INT8 tensor it emits. Written by make_calibration.py "
                   "from the oracle's fp64 real-valued model.", "configs": {}}
    for name in ("cfg0", "cfg1", "cfg2", "cfg3"):
        cfg = C.CONFIGS[name]
        chains = {}
        for ch in cfg.chains:
            x = C.chain_input(ch)
            params = C.chain_params(ch)
            first_wh = ch.s_in if (ch.layers[0].form == C.WH and ch.input_kind == "i8") else None
            scales = O.calibrate_chain(ch.layers, params, real_input(ch, x), first_wh)
            chains[ch.name] = scales
            print(name, ch.name, [(round(s["s_x"], 5), round(s["s_out"], 5)) for s in scales], flush=True)
        out["configs"][name] = chains
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "calibration.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
    print("wrote", path)


if __name__ == "__main__":
    main()
