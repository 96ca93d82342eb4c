"""Fit the Zipf router-bias scale of the large_zipf_bf16 workload with the oracle.

TEST INFRASTRUCTURE (calls only oracle/ and synth/). The workload wants expert
popularity close to Zipf(s=1.2): the share of (token, pick) pairs of the expert of
rank r should be close to r^-1.2 / sum_r' r'^-1.2. The bias is b_e = -c s ln(rank_e);
this script bisects c on the L1 distance between the realised shares (oracle routing
of the seeded tokens) and the target shares, and prints c and the shares. The value
is copied by hand into synth/moe_inputs.py as ZIPF_BIAS_SCALE.

Usage: python -m oracle.calibrate_zipf [--tokens N]
"""
import argparse

import numpy as np

from synth import moe_inputs as mi
from oracle import moe_oracle as mo


def shares_for(c, x, wr, ranks, s, k):
    b = (-c * s * np.log(ranks.astype(np.float64)))[None, :]
    z = mo.router_logits(x, wr, b, [0, x.shape[0]])
    idx = mo.topk_indices(z.astype(np.float32), k)
    counts = np.bincount(idx.ravel(), minlength=wr.shape[1]).astype(np.float64)
    order = np.argsort(ranks)  # experts by rank 1..E
    return counts[order] / counts.sum()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--tokens", type=int, default=4096)
    a = ap.parse_args()
    shape = mi.SHAPES[4]
    inp = mi.make_inputs(shape, with_weights=False)
    x = inp["x"][: a.tokens]
    ranks = inp["zipf_rank"]
    E, s, k = shape.n_experts, shape.zipf_s, shape.top_k
    target = np.arange(1, E + 1, dtype=np.float64) ** (-s)
    target /= target.sum()

    def dist(c):
        return np.abs(shares_for(c, x, inp["w_router"], ranks, s, k) - target).sum()

    lo, hi = 0.0, 8.0
    for _ in range(30):  # golden-section search on a unimodal distance
        m1, m2 = lo + (hi - lo) * 0.382, lo + (hi - lo) * 0.618
        if dist(m1) < dist(m2):
            hi = m2
        else:
            lo = m1
    c = round(0.5 * (lo + hi), 3)
    print("ZIPF_BIAS_SCALE =", c)
    print("target  ", np.round(target, 3))
    print("realised", np.round(shares_for(c, x, inp["w_router"], ranks, s, k), 3))


if __name__ == "__main__":
    main()
