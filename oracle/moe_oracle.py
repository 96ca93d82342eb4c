"""fp64 CPU oracle of the sparse MoE expert layer, forward and backward.

TEST INFRASTRUCTURE ONLY. Only tests/, ``__graft_entry__.smoke()`` and the CPU
baseline legs of ``bench.py`` may import this module. The product path (the CUDA
library and its Python binding) never imports, calls or links anything here, and
nothing here imports the product path. Inputs come from ``synth`` only.

What it computes (PC-MoE, arXiv 2506.02965):
  * Gating, Alg. 7: p = Softmax(W_i h); I = TopKIndices(p); w = p[I]
    (no renormalisation; ``normalize_topk=1`` is the common renormalised variant).
  * ProcessExperts, Alg. 3: h^e = sum_{idx in I} w[idx] * E_idx(h). The "send h to
    the host of idx" step becomes the expert-major permutation below.
  * ForwardExpert / BackwardExpert, Alg. 6: E_j(h) and back-propagation through E_j.
  * BackwardExperts, Alg. 5 with the chain rule written out in full: each expert
    receives w * dOut, and the gate weights receive <dOut, E_idx(h)>.
  * Section 3.2 ("Backward propagation"): the expert host gets the gradient w.r.t.
    the expert output and returns one activation-sized gradient w.r.t. its input.

Readings where the paper is silent:
  R1 expert = SwiGLU, E(h) = W2 (silu(W1g h) * (W1u h)), W1 = [W1g; W1u] of shape
     [2F, d] (gate rows first), no biases, no capacity limit;
  R2 optional router bias b (absent unless given);
  R3 top-k decided on fp32 logits (the kernel's precision), descending, ties to the
     lower expert id; the selection is a constant in the backward;
  R4 permutation is expert-major and stable (ascending token id inside an expert);
  R5 aux loss (Switch form) L_p = alpha * E * sum_e f_pe * P_pe per party,
     f_pe = counts_pe / (T_p k) (no gradient), P_pe = mean_{t in p} p_te;
  R6 shared experts are dense SwiGLU experts on every token, added with weight 1;
  R7 party p owns tokens [po[p], po[p+1]) and routes them with its own W_r[p], b[p].

Everything is float64 numpy. A library matmul serves as the row-wise dot product;
no other blocking, fusion or reordering is done.
"""
from __future__ import annotations

import numpy as np

f64 = np.float64


# ----------------------------------------------------------------------------- gating

def party_of_tokens(T: int, party_offsets) -> np.ndarray:
    """Party index of each token (R7)."""
    po = np.asarray(party_offsets, dtype=np.int64)
    part = np.empty(T, dtype=np.int64)
    for p in range(len(po) - 1):
        part[po[p]:po[p + 1]] = p
    return part


def router_logits(x, w_router, router_bias, party_offsets) -> np.ndarray:
    """z_t = W_{p(t)} h_t (+ b_{p(t)}): the argument of Softmax in Alg. 7 (R2, R7)."""
    x = np.asarray(x, f64)
    W = np.asarray(w_router, f64)  # [P, E, d]
    po = np.asarray(party_offsets, dtype=np.int64)
    z = np.empty((x.shape[0], W.shape[1]), f64)
    for p in range(W.shape[0]):
        rows = slice(po[p], po[p + 1])
        z[rows] = x[rows] @ W[p].T
        if router_bias is not None:
            z[rows] += np.asarray(router_bias, f64)[p]
    return z


def softmax(z) -> np.ndarray:
    """p = Softmax(z) along experts (Alg. 7), max-subtracted."""
    z = np.asarray(z, f64)
    e = np.exp(z - z.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


def topk_indices(z32, k: int) -> np.ndarray:
    """TopKIndices of Alg. 7, decided on fp32 logits (R3).

    Softmax is monotone, so ranking p and ranking z agree. Order: descending
    logit, equal logits ordered by ascending expert id.
    """
    z32 = np.asarray(z32, np.float32)
    T, E = z32.shape
    idx = np.empty((T, k), np.int32)
    for t in range(T):
        order = sorted(range(E), key=lambda e: (-float(z32[t, e]), e))
        idx[t] = order[:k]
    return idx


def gate_weights(p, idx, normalize_topk: int = 0) -> np.ndarray:
    """w = p[I] (Alg. 7); renormalised over the k picks when normalize_topk=1."""
    p = np.asarray(p, f64)
    w = np.take_along_axis(p, idx.astype(np.int64), axis=1)
    if normalize_topk:
        w = w / w.sum(axis=1, keepdims=True)
    return w


def top_margin(z, k: int) -> np.ndarray:
    """Per token, the smallest gap between neighbouring logits among the top k+1.

    A token whose margin exceeds twice the logit error of a computation is routed
    the same way, in the same order, by any computation within that error.
    """
    zs = -np.sort(-np.asarray(z, f64), axis=1)
    kk = min(k + 1, zs.shape[1])
    if kk < 2:
        return np.full(zs.shape[0], np.inf)
    return np.min(zs[:, :kk - 1] - zs[:, 1:kk], axis=1)


# ----------------------------------------------------------------------------- dispatch

def dispatch_tables(idx, n_experts: int):
    """Per-expert counts, prefix offsets and the stable expert-major permutation (R4).

    counts_e   = #{(t, j) : I_tj = e}
    offsets_e  = sum_{e' < e} counts_e'            (offsets_E = T k)
    slot(t, j) = offsets_{I_tj} + #{t' < t : I_tj in I_t'}
    token_of[slot(t, j)] = t
    """
    idx = np.asarray(idx)
    T, k = idx.shape
    counts = np.zeros(n_experts, np.int64)
    for t in range(T):
        for j in range(k):
            counts[idx[t, j]] += 1
    offsets = np.zeros(n_experts + 1, np.int64)
    for e in range(n_experts):
        offsets[e + 1] = offsets[e] + counts[e]
    seen = np.zeros(n_experts, np.int64)  # tokens t' < t that picked e
    slot_of = np.empty((T, k), np.int64)
    for t in range(T):
        for j in range(k):
            e = idx[t, j]
            slot_of[t, j] = offsets[e] + seen[e]
        for j in range(k):
            seen[idx[t, j]] += 1
    token_of = np.empty(T * k, np.int64)
    for t in range(T):
        for j in range(k):
            token_of[slot_of[t, j]] = t
    return counts, offsets, slot_of, token_of


def owner_of(e: int, n_parties: int) -> int:
    """The party hosting expert e: round-robin over the parties (Sec. 3.1 item 2; R7)."""
    return e % n_parties


def owner_dispatch_tables(idx, n_experts: int, party_offsets):
    """The dispatch grouped by receiving party: the layout of the cross-party sends of
    Alg. 3 ("send h to the host of idx") when expert e lives on party owner(e).

    group_expert[g] = the g-th expert in (owner, expert) order
    counts_g, offsets_g, slot(t, j), token_of as dispatch_tables, with the expert
      segments in that order: slot(t, j) = offsets_{pos(I_tj)} + #{t' < t : I_tj in I_t'}
    send[s, o] = #{(t, j) : t in party s, owner(I_tj) = o}  (sends from s received by o;
      tokens are party-contiguous, so inside a segment the rows of each source party are
      contiguous and in party order)
    """
    idx = np.asarray(idx)
    T, k = idx.shape
    po = np.asarray(party_offsets, dtype=np.int64)
    P = len(po) - 1
    group_expert = sorted(range(n_experts), key=lambda e: (owner_of(e, P), e))
    pos = np.empty(n_experts, np.int64)
    for g, e in enumerate(group_expert):
        pos[e] = g
    counts = np.zeros(n_experts, np.int64)  # per segment g
    for t in range(T):
        for j in range(k):
            counts[pos[idx[t, j]]] += 1
    offsets = np.zeros(n_experts + 1, np.int64)
    for g in range(n_experts):
        offsets[g + 1] = offsets[g] + counts[g]
    seen = np.zeros(n_experts, np.int64)
    slot_of = np.empty((T, k), np.int64)
    for t in range(T):
        for j in range(k):
            g = pos[idx[t, j]]
            slot_of[t, j] = offsets[g] + seen[g]
        for j in range(k):
            seen[pos[idx[t, j]]] += 1
    token_of = np.empty(T * k, np.int64)
    for t in range(T):
        for j in range(k):
            token_of[slot_of[t, j]] = t
    send = np.zeros((P, P), np.int64)
    party = party_of_tokens(T, po)
    for t in range(T):
        for j in range(k):
            send[party[t], owner_of(idx[t, j], P)] += 1
    return np.asarray(group_expert, np.int64), counts, offsets, slot_of, token_of, send


def party_counts(idx, n_experts: int, party_offsets) -> np.ndarray:
    """counts_{p,e}: how many of party p's (token, pick) pairs went to expert e."""
    po = np.asarray(party_offsets, dtype=np.int64)
    P = len(po) - 1
    c = np.zeros((P, n_experts), np.int64)
    for p in range(P):
        for t in range(po[p], po[p + 1]):
            for e in idx[t]:
                c[p, e] += 1
    return c


def gather_permute(x, token_of):
    """x_perm[r] = x[token_of[r]]: each token's hidden state "sent" to every expert
    it picked (Alg. 3, Send h to the host of idx), laid out expert-major."""
    x = np.asarray(x, f64)
    x_perm = np.empty((len(token_of), x.shape[1]), f64)
    for r, t in enumerate(token_of):
        x_perm[r] = x[t]
    return x_perm


def combine(y_perm, w, slot_of):
    """h^e_t = sum_j w_tj * E_{I_tj}(h_t) (Alg. 3, the weighted sum returned to P_i)."""
    T, k = slot_of.shape
    out = np.zeros((T, y_perm.shape[1]), f64)
    for t in range(T):
        for j in range(k):
            out[t] += w[t, j] * y_perm[slot_of[t, j]]
    return out


def combine_backward(dout, y_perm, w, slot_of):
    """Chain rule of the weighted sum: dY at slot(t,j) = w_tj dOut_t (the gradient each
    expert host receives, Alg. 5 / Sec. 3.2) and dw_tj = <dOut_t, E_{I_tj}(h_t)>."""
    T, k = slot_of.shape
    dout = np.asarray(dout, f64)
    dy_perm = np.zeros((T * k, dout.shape[1]), f64)
    dw = np.zeros((T, k), f64)
    for t in range(T):
        for j in range(k):
            r = slot_of[t, j]
            dy_perm[r] = w[t, j] * dout[t]
            dw[t, j] = np.dot(dout[t], y_perm[r])
    return dy_perm, dw


def unpermute_reduce(dx_perm, slot_of):
    """dx_t = sum_j dXp[slot(t,j)]: the activation-sized input gradients the expert
    hosts return to the data owner (Sec. 3.2), summed per token."""
    T, k = slot_of.shape
    dx = np.zeros((T, dx_perm.shape[1]), f64)
    for t in range(T):
        for j in range(k):
            dx[t] += dx_perm[slot_of[t, j]]
    return dx


# ----------------------------------------------------------------------------- experts

def silu(g):
    return g / (1.0 + np.exp(-g))


def sigmoid(g):
    return 1.0 / (1.0 + np.exp(-g))


def swiglu_forward(X, W1e, W2e):
    """E(h) of Alg. 6 under R1: returns G, U, A = silu(G)*U and Y = A W2^T."""
    X = np.asarray(X, f64)
    W1e = np.asarray(W1e, f64)
    W2e = np.asarray(W2e, f64)
    F = W1e.shape[0] // 2
    G = X @ W1e[:F].T
    U = X @ W1e[F:].T
    A = silu(G) * U
    Y = A @ W2e.T
    return G, U, A, Y


def swiglu_backward(X, W1e, W2e, G, U, A, dY):
    """Back-propagation through one SwiGLU expert (Alg. 6, BackwardExpert).

    dA = dY W2;  dU = dA * silu(G);  dG = dA * U * s (1 + G (1 - s)), s = sigmoid(G);
    dW2 = dY^T A;  dW1 = [dG | dU]^T X;  dX = [dG | dU] W1.
    """
    X = np.asarray(X, f64)
    W1e = np.asarray(W1e, f64)
    W2e = np.asarray(W2e, f64)
    dA = dY @ W2e
    s = sigmoid(G)
    dU = dA * (G * s)
    dG = dA * U * s * (1.0 + G * (1.0 - s))
    dH = np.concatenate([dG, dU], axis=1)
    dW2 = dY.T @ A
    dW1 = dH.T @ X
    dX = dH @ W1e
    return dH, dX, dW1, dW2


# ----------------------------------------------------------------------------- aux loss

def aux_loss(probs, counts_pe, party_offsets, k: int, alpha: float):
    """Load-balancing loss per party (R5) and its gradient coefficient.

    L_p = alpha * E * sum_e f_pe * P_pe, f_pe = counts_pe / (T_p k),
    P_pe = (1/T_p) sum_{t in p} p_te.  dL_p/dp_te = alpha * E * f_pe / T_p for t in p.
    """
    probs = np.asarray(probs, f64)
    po = np.asarray(party_offsets, dtype=np.int64)
    P, E = counts_pe.shape
    loss = np.zeros(P, f64)
    coef = np.zeros((P, E), f64)
    for p in range(P):
        Tp = po[p + 1] - po[p]
        f = counts_pe[p] / (Tp * k)
        Pm = probs[po[p]:po[p + 1]].sum(axis=0) / Tp
        loss[p] = alpha * E * np.sum(f * Pm)
        coef[p] = alpha * E * f / Tp
    return loss, coef


# ----------------------------------------------------------------------------- layer

def layer_forward(inp: dict, shape) -> dict:
    """Forward of the MoE layer (Alg. 7 then Alg. 3 with Alg. 6 experts)."""
    T, E, k = shape.T, shape.n_experts, shape.top_k
    x = np.asarray(inp["x"], f64)
    po = inp["party_offsets"]
    z = router_logits(x, inp["w_router"], inp.get("router_bias"), po)
    z32 = z.astype(np.float32)
    p = softmax(z)
    idx = topk_indices(z32, k)
    w = gate_weights(p, idx, shape.normalize_topk)
    counts, offsets, slot_of, token_of = dispatch_tables(idx, E)
    cpe = party_counts(idx, E, po)
    x_perm = gather_permute(x, token_of)
    F = shape.d_ff
    h_gu = np.zeros((T * k, 2 * F), f64)
    act = np.zeros((T * k, F), f64)
    y_perm = np.zeros((T * k, shape.d_model), f64)
    for e in range(E):
        r = slice(offsets[e], offsets[e + 1])
        if offsets[e + 1] == offsets[e]:
            continue
        G, U, A, Y = swiglu_forward(x_perm[r], inp["w1"][e], inp["w2"][e])
        h_gu[r, :F], h_gu[r, F:], act[r], y_perm[r] = G, U, A, Y
    out = combine(y_perm, w, slot_of)
    shared = []
    for s in range(shape.n_shared):
        G, U, A, Y = swiglu_forward(x, inp["ws1"][s], inp["ws2"][s])
        shared.append((G, U, A, Y))
        out += Y
    loss, coef = aux_loss(p, cpe, po, k, shape.aux_alpha)
    return dict(logits=z, logits32=z32, probs=p, topk_idx=idx, topk_w=w,
                counts=counts, party_counts=cpe, offsets=offsets, slot_of=slot_of,
                token_of=token_of, x_perm=x_perm, h_gu=h_gu, act=act, y_perm=y_perm,
                out=out, shared=shared, aux_loss=loss, aux_coef=coef)


def layer_backward(inp: dict, shape, fwd: dict, dout=None, with_aux: bool = True) -> dict:
    """Backward of the MoE layer: Alg. 5 and Alg. 6 with the chain rule completed."""
    T, E, k, F = shape.T, shape.n_experts, shape.top_k, shape.d_ff
    d = shape.d_model
    x = np.asarray(inp["x"], f64)
    dout = np.asarray(inp["dout"] if dout is None else dout, f64)
    idx, w, p = fwd["topk_idx"], fwd["topk_w"], fwd["probs"]
    slot_of, offsets = fwd["slot_of"], fwd["offsets"]
    y_perm = fwd["y_perm"]
    dy_perm, dw = combine_backward(dout, y_perm, w, slot_of)
    # experts
    dh = np.zeros((T * k, 2 * F), f64)
    dx_perm = np.zeros((T * k, d), f64)
    dw1 = np.zeros((E, 2 * F, d), f64)
    dw2 = np.zeros((E, d, F), f64)
    for e in range(E):
        r = slice(offsets[e], offsets[e + 1])
        if offsets[e + 1] == offsets[e]:
            continue
        G, U = fwd["h_gu"][r, :F], fwd["h_gu"][r, F:]
        dH, dX, dW1, dW2 = swiglu_backward(fwd["x_perm"][r], inp["w1"][e], inp["w2"][e],
                                           G, U, fwd["act"][r], dy_perm[r])
        dh[r], dx_perm[r], dw1[e], dw2[e] = dH, dX, dW1, dW2
    shared_grads = []
    dx_shared = np.zeros((T, d), f64)
    for s in range(shape.n_shared):
        G, U, A, _ = fwd["shared"][s]
        dH, dX, dW1, dW2 = swiglu_backward(x, inp["ws1"][s], inp["ws2"][s], G, U, A, dout)
        shared_grads.append((dH, dX, dW1, dW2))
        dx_shared += dX
    # gate weights -> probabilities
    dp = np.zeros((T, E), f64)
    if shape.normalize_topk:
        psel = np.take_along_axis(p, idx.astype(np.int64), axis=1)
        S = psel.sum(axis=1)
        inner = (dw * w).sum(axis=1)
        for t in range(T):
            for j in range(k):
                dp[t, idx[t, j]] += (dw[t, j] - inner[t]) / S[t]
    else:
        for t in range(T):
            for j in range(k):
                dp[t, idx[t, j]] += dw[t, j]
    po = np.asarray(inp["party_offsets"], dtype=np.int64)
    part = party_of_tokens(T, po)
    if with_aux:
        dp += fwd["aux_coef"][part]
    # softmax backward
    dz = p * (dp - np.sum(dp * p, axis=1, keepdims=True))
    Wr = np.asarray(inp["w_router"], f64)
    P = Wr.shape[0]
    dw_router = np.zeros_like(Wr)
    dbias = np.zeros((P, E), f64)
    dx_router = np.zeros((T, d), f64)
    for q in range(P):
        rows = slice(po[q], po[q + 1])
        dw_router[q] = dz[rows].T @ x[rows]
        dbias[q] = dz[rows].sum(axis=0)
        dx_router[rows] = dz[rows] @ Wr[q]
    dx = unpermute_reduce(dx_perm, slot_of) + dx_router + dx_shared
    return dict(dy_perm=dy_perm, dtopk_w=dw, dh=dh, dx_perm=dx_perm, dw1=dw1, dw2=dw2,
                dprobs=dp, dlogits=dz, dw_router=dw_router, dbias=dbias, dx=dx,
                shared_grads=shared_grads, dx_router=dx_router)


def router_backward(inp: dict, shape, probs, idx, topk_w, dtopk_w, aux_coef=None) -> dict:
    """Backward of the gating function alone (Alg. 7; the router is trained as part of
    the party's local layers, Sec. 3.1) for given picks I, gate weights w and their
    gradients dw, with the picks held constant (R3):

      dp_te = sum_j [I_tj = e] g_tj + dL_aux/dp_te,
              g_tj = dw_tj, or (dw_tj - <dw_t, w_t>) / sum_j p_{t,I_tj} when renormalised;
      dz_t  = p_t * (dp_t - <dp_t, p_t>)                  (softmax backward)
      dW_r[q] = sum_{t in q} dz_t^T x_t;  db[q] = sum_{t in q} dz_t;  dx_router,t = dz_t W_r[q(t)]

    The same steps as the router part of layer_backward, written for any picks: it needs
    no expert output, so it runs at every workload size.
    """
    T, E, k = shape.T, shape.n_experts, shape.top_k
    p = np.asarray(probs, f64)
    idx = np.asarray(idx)
    w = np.asarray(topk_w, f64)
    dw = np.asarray(dtopk_w, f64)
    dp = np.zeros((T, E), f64)
    if shape.normalize_topk:
        psel = np.take_along_axis(p, idx.astype(np.int64), axis=1)
        S = psel.sum(axis=1)
        inner = (dw * w).sum(axis=1)
        for t in range(T):
            for j in range(k):
                dp[t, idx[t, j]] += (dw[t, j] - inner[t]) / S[t]
    else:
        for t in range(T):
            for j in range(k):
                dp[t, idx[t, j]] += dw[t, j]
    po = np.asarray(inp["party_offsets"], dtype=np.int64)
    part = party_of_tokens(T, po)
    if aux_coef is not None:
        dp += np.asarray(aux_coef, f64)[part]
    dz = p * (dp - np.sum(dp * p, axis=1, keepdims=True))
    x = np.asarray(inp["x"], f64)
    Wr = np.asarray(inp["w_router"], f64)
    P = Wr.shape[0]
    dw_router = np.zeros_like(Wr)
    dbias = np.zeros((P, E), f64)
    dx_router = np.zeros((T, shape.d_model), f64)
    for q in range(P):
        rows = slice(po[q], po[q + 1])
        dw_router[q] = dz[rows].T @ x[rows]
        dbias[q] = dz[rows].sum(axis=0)
        dx_router[rows] = dz[rows] @ Wr[q]
    return dict(dprobs=dp, dlogits=dz, dw_router=dw_router, dbias=dbias, dx_router=dx_router)


# ----------------------------------------------------------------------------- sampled

def route_all(inp: dict, shape) -> dict:
    """Routing of every token (cheap at any size): logits, probs, picks, counts, aux."""
    T, E, k = shape.T, shape.n_experts, shape.top_k
    po = inp["party_offsets"]
    z = router_logits(inp["x"], inp["w_router"], inp.get("router_bias"), po)
    z32 = z.astype(np.float32)
    p = softmax(z)
    idx = topk_indices(z32, k)
    w = gate_weights(p, idx, shape.normalize_topk)
    cpe = party_counts(idx, E, po)
    loss, coef = aux_loss(p, cpe, po, k, shape.aux_alpha)
    return dict(logits=z, logits32=z32, probs=p, topk_idx=idx, topk_w=w,
                party_counts=cpe, counts=cpe.sum(axis=0), aux_loss=loss, aux_coef=coef)


def sampled_token_rows(inp: dict, shape, route: dict, tokens) -> dict:
    """Per-token outputs of the full layer for a few tokens, one token at a time.

    The same definitions as layer_forward/layer_backward restricted to the given
    tokens: out_t, dw_t (gate grads), dz_t (logit grads), dx_t, and for each pick j
    the expert output Y_tj and the expert input gradient dXp_tj.
    """
    k, F = shape.top_k, shape.d_ff
    x = np.asarray(inp["x"], f64)
    dout = np.asarray(inp["dout"], f64)
    part = party_of_tokens(shape.T, inp["party_offsets"])
    Wr = np.asarray(inp["w_router"], f64)
    res = {n: [] for n in ("out", "dtopk_w", "dlogits", "dx", "y", "dx_perm")}
    for t in tokens:
        xt = x[t:t + 1]
        e_list = route["topk_idx"][t]
        w = route["topk_w"][t]
        p = route["probs"][t]
        out = np.zeros(shape.d_model, f64)
        dx = np.zeros(shape.d_model, f64)
        ys, dxps, dw = [], [], np.zeros(k, f64)
        for j, e in enumerate(e_list):
            G, U, A, Y = swiglu_forward(xt, inp["w1"][e], inp["w2"][e])
            out += w[j] * Y[0]
            dw[j] = np.dot(dout[t], Y[0])
            _, dX, _, _ = swiglu_backward(xt, inp["w1"][e], inp["w2"][e], G, U, A,
                                          w[j] * dout[t:t + 1])
            ys.append(Y[0])
            dxps.append(dX[0])
            dx += dX[0]
        for s in range(shape.n_shared):
            G, U, A, Y = swiglu_forward(xt, inp["ws1"][s], inp["ws2"][s])
            out += Y[0]
            _, dX, _, _ = swiglu_backward(xt, inp["ws1"][s], inp["ws2"][s], G, U, A,
                                          dout[t:t + 1])
            dx += dX[0]
        dp = np.zeros(shape.n_experts, f64)
        if shape.normalize_topk:
            S = p[e_list].sum()
            inner = np.dot(dw, w)
            for j, e in enumerate(e_list):
                dp[e] += (dw[j] - inner) / S
        else:
            for j, e in enumerate(e_list):
                dp[e] += dw[j]
        dp += route["aux_coef"][part[t]]
        dz = p * (dp - np.dot(dp, p))
        dx += dz @ Wr[part[t]]
        for n, v in (("out", out), ("dtopk_w", dw), ("dlogits", dz), ("dx", dx),
                     ("y", np.stack(ys)), ("dx_perm", np.stack(dxps))):
            res[n].append(v)
    return {n: np.stack(v) for n, v in res.items()}


def sampled_weight_grads(inp: dict, shape, route: dict, e: int, f_cols) -> dict:
    """Selected slices of dW1[e] and dW2[e], summed over every token routed to e.

    dW2[e][:, f] = sum_t dY_t A_t[f];  dW1[e][f, :] and dW1[e][F+f, :] =
    sum_t dG_t[f] x_t and sum_t dU_t[f] x_t, with dY_t = w_tj dOut_t.
    Only column f of G, U and dA is needed, so each slice costs O(M_e d).
    """
    F = shape.d_ff
    x = np.asarray(inp["x"], f64)
    dout = np.asarray(inp["dout"], f64)
    idx, w = route["topk_idx"], route["topk_w"]
    toks, ws = [], []
    for t in range(shape.T):
        for j in range(shape.top_k):
            if idx[t, j] == e:
                toks.append(t)
                ws.append(w[t, j])
    toks = np.asarray(toks, np.int64)
    Xe = x[toks]
    dYe = dout[toks] * np.asarray(ws, f64)[:, None]
    W1e = np.asarray(inp["w1"][e], f64)
    W2e = np.asarray(inp["w2"][e], f64)
    dw2_cols, dw1_gate_rows, dw1_up_rows = [], [], []
    for f in f_cols:
        G = Xe @ W1e[f]
        U = Xe @ W1e[F + f]
        s = sigmoid(G)
        A = G * s * U
        dA = dYe @ W2e[:, f]
        dU = dA * G * s
        dG = dA * U * s * (1.0 + G * (1.0 - s))
        dw2_cols.append(dYe.T @ A)
        dw1_gate_rows.append(dG @ Xe)
        dw1_up_rows.append(dU @ Xe)
    return dict(dw2_cols=np.stack(dw2_cols, axis=1),
                dw1_gate_rows=np.stack(dw1_gate_rows),
                dw1_up_rows=np.stack(dw1_up_rows), n_rows=len(toks))
