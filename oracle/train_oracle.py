"""fp64 CPU oracle of PC-MoE's sequential collaborative training (Alg. 1) on a toy block.

TEST INFRASTRUCTURE ONLY. Only tests/ may import this module; the product path never
imports, calls or links anything here, and nothing here imports the product path.
Inputs (initial parameters, data, the turn order) come from ``synth`` only.

What it computes. Alg. 1 (sequential version): in every epoch the parties take turns
in a random order; party i processes B batches of its own data; per batch it runs
LocalForward (Alg. 2) whose one expert step is ProcessExperts (Alg. 3) with its own
gating G_i (Alg. 7) over the shared expert pool, takes the loss, back-propagates
through its local layers and updates them (BackwardLocal, Alg. 4), and sends the
gradient to the experts it called, which update themselves (BackwardExperts and
BackwardExpert, Alg. 5 and 6). Nothing else changes: no global broadcast.

Readings where the paper leaves the toy open:
  T1 the block is one expert step and nothing else: h = ProcessExperts(x, P_i, G_i);
     the gating W_r[i] is party i's only local layer (the backbone is out of scope);
  T2 Loss(h, y) = sum_t ||h_t - y_t||^2 / (2T) (regression on synthetic targets) plus
     the layer's load-balancing loss (alpha of the shape), both back-propagated;
  T3 the update is plain SGD, w <- w - lr * dL/dw, right after each batch's backward;
  T4 the experts "called" by a batch are those with at least one routed token; an
     expert with none keeps its parameters bit for bit (its gradient is zero anyway);
  T5 a batch holds one party's tokens only; D_i is read in order and cycled;
  T6 the parties hosting called experts are {e mod n} (round-robin ownership).

Everything is float64 numpy on top of ``moe_oracle``'s layer forward and backward.
"""
from __future__ import annotations

import numpy as np

from oracle import moe_oracle as mo

f64 = np.float64


def mse_loss(out, y):
    """Loss(h, y) of T2 without the aux term and its gradient dL/dh = (h - y) / T."""
    out = np.asarray(out, f64)
    y = np.asarray(y, f64)
    T = out.shape[0]
    diff = out - y
    return float(np.sum(diff * diff) / (2.0 * T)), diff / T


def sgd_groups(w, dw, lr: float, counts=None):
    """One SGD step (T3) on a parameter stacked as groups along axis 0: group g moves
    by -lr * dw[g] when counts is None or counts[g] > 0, else keeps its values (T4)."""
    w = np.asarray(w, f64)
    dw = np.asarray(dw, f64)
    new = w - f64(lr) * dw
    if counts is not None:
        keep = np.asarray(counts) <= 0
        new[keep] = w[keep]
    return new


def _layer_inputs(params, party: int, x):
    T = x.shape[0]
    return {"x": np.asarray(x, f64), "w_router": np.asarray(params["w_router"], f64)[party:party + 1],
            "router_bias": None, "party_offsets": np.array([0, T], np.int64),
            "w1": np.asarray(params["w1"], f64), "w2": np.asarray(params["w2"], f64),
            "ws1": None, "ws2": None}


def batch_loss(params, party: int, x, y, shape):
    """The objective of one batch under T1/T2 (MSE plus aux loss) and the forward pass."""
    fwd = mo.layer_forward(_layer_inputs(params, party, x), shape)
    mse, dout = mse_loss(fwd["out"], y)
    return mse + float(fwd["aux_loss"][0]), mse, dout, fwd


def train_step(params, party: int, x, y, shape, lr: float):
    """One batch of Alg. 1's inner loop for party ``party``: forward, loss, backward,
    the router update (BackwardLocal) and the called experts' updates (BackwardExpert).
    ``shape`` describes the batch (T tokens, one party). Returns the new parameters
    and a record: total loss, MSE, aux loss, per-expert counts, the smallest top-(k+1)
    logit gap of the batch, gradients, updated parties."""
    inp = _layer_inputs(params, party, x)
    loss, mse, dout, fwd = batch_loss(params, party, x, y, shape)
    bwd = mo.layer_backward(inp, shape, fwd, dout=dout, with_aux=True)
    counts = np.asarray(fwd["counts"])
    new = {k: np.array(v, f64) for k, v in params.items()}
    new["w_router"][party] = sgd_groups(params["w_router"][party:party + 1], bwd["dw_router"], lr)[0]
    new["w1"] = sgd_groups(params["w1"], bwd["dw1"], lr, counts)
    new["w2"] = sgd_groups(params["w2"], bwd["dw2"], lr, counts)
    n = np.asarray(params["w_router"]).shape[0]
    owners = {int(e) % n for e in np.nonzero(counts > 0)[0]}
    rec = {"party": party, "loss": loss, "mse": mse, "aux": float(fwd["aux_loss"][0]), "counts": counts,
           "min_margin": float(mo.top_margin(fwd["logits"], shape.top_k).min()),
           "dw_router": bwd["dw_router"][0], "dw1": bwd["dw1"], "dw2": bwd["dw2"],
           "updated_parties": sorted(owners | {party})}
    return new, rec


def round_robin_train(params, batches, schedule, B: int, shape, lr: float):
    """Alg. 1: for each epoch's permutation in ``schedule``, each party in that order
    processes B batches of its data ``batches[i]`` (T5: read in order, cycled), one
    ``train_step`` each. Returns the final parameters and one record per batch (with
    the batch index used)."""
    params = {k: np.array(v, f64) for k, v in params.items()}
    used = [0] * len(batches)
    log = []
    for order in schedule:
        for i in order:
            for _ in range(B):
                b = used[i] % len(batches[i])
                used[i] += 1
                x, y = batches[i][b]
                params, rec = train_step(params, i, x, y, shape, lr)
                rec["batch"] = b
                log.append(rec)
    return params, log
