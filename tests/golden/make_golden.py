"""Write the stored expected values under tests/golden/ (run by hand after a deliberate
change of the oracle's arithmetic; the commit that does so names the passage that
justifies it).

The paper prints no numeric example of the layer or of its training protocol, so these
values come from the fp64 oracle on small seeded inputs (this script calls only
``oracle/`` and ``synth/``). They pin the oracle against unintended change; what pins
it against the paper are the closed forms, invariants, brute force and finite
differences of tests/test_oracle_pins.py and tests/test_train_oracle_pins.py.

    python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import moe_oracle as mo  # noqa: E402
from oracle import train_oracle as to  # noqa: E402
from synth import moe_inputs as mi  # noqa: E402

LAYER = mi.MoEShape("golden_layer", T=12, d_model=8, n_experts=4, d_ff=6, top_k=2, dtype="f32",
                    n_parties=2, n_shared=1, d_ff_shared=4, aux_alpha=0.5, seed=4242)
TRAIN = mi.MoEShape("golden_train", T=8, d_model=8, n_experts=4, d_ff=6, top_k=2, dtype="f32",
                    aux_alpha=0.1, seed=4343)


def layer_values():
    inp = mi.make_inputs(LAYER)
    fwd = mo.layer_forward(inp, LAYER)
    bwd = mo.layer_backward(inp, LAYER, fwd)
    return {"topk_idx": fwd["topk_idx"].tolist(), "offsets": np.asarray(fwd["offsets"]).tolist(),
            "out": fwd["out"].tolist(), "aux_loss": np.asarray(fwd["aux_loss"]).tolist(),
            "dx": bwd["dx"].tolist(), "dw_router": bwd["dw_router"].tolist(),
            "dw1_sum_per_expert": bwd["dw1"].sum(axis=(1, 2)).tolist(),
            "dw2_sum_per_expert": bwd["dw2"].sum(axis=(1, 2)).tolist()}


def train_values():
    n, B = 3, 2
    init = mi.train_init(TRAIN, n, seed=TRAIN.seed)
    batches = mi.train_batches(TRAIN, n, 2, seed=TRAIN.seed + 1)
    sched = mi.party_schedule(n, 2, seed=TRAIN.seed + 2)
    final, log = to.round_robin_train(init, batches, sched, B, TRAIN, 0.05)
    return {"schedule": sched, "order": [[r["party"], r["batch"]] for r in log],
            "loss": [r["loss"] for r in log],
            "w_router_sum_per_party": final["w_router"].sum(axis=(1, 2)).tolist(),
            "w1_sum_per_expert": final["w1"].sum(axis=(1, 2)).tolist()}


def main():
    for name, fn in (("layer_tiny.json", layer_values), ("train_tiny.json", train_values)):
        with open(os.path.join(HERE, name), "w") as f:
            json.dump({"source": "fp64 oracle (oracle/), inputs from synth/; written by make_golden.py",
                       "values": fn()}, f, indent=1)


if __name__ == "__main__":
    main()
