"""fp64 oracle of the character-LM block around the mixing stack.

TEST INFRASTRUCTURE, NOT PRODUCT CODE: only the test suite, the smoke check
and the CPU-baseline leg of the benchmark import this module.  The CUDA path
never does, and this module imports nothing from the CUDA path.

The block (App. A: width d, hidden 1024 = 2d at d = 512; the weight counts of
Table B2ecost / B1cost fit exactly token and position embeddings, two
LayerNorms and an FFN with biases per layer, a final LayerNorm and an output
head with bias).  Readings where the paper is silent: pre-norm residual
sublayers, ReLU in the FFN, no bias on the mixing maps, LayerNorm with the
biased variance and eps = 1e-5, next-symbol cross-entropy averaged over the
B n positions:

    x = E[ids[:, :n]] + P
    for layer l (rotated schedule, cube dimension l mod log2 n, causal):
        h = LN1_l(x);   x = x + M_l(h)            M_l: Eq. (1), no bias
        g = LN2_l(x);   u = g W1_l^T + b1_l;   x = x + relu(u) W2_l^T + b2_l
    hf = LNf(x);   logits = hf Wh^T + bh
    loss = mean over (b, t) of logsumexp(logits[b, t]) - logits[b, t, ids[b, t + 1]]

The mixing sublayer M_l is the oracle's layer of Eq. (1) (``oracle.layer_fwd``
/ ``layer_bwd``); everything else is written out here with numpy in fp64.

``round_bf16=True`` rounds to bfloat16 exactly the tensors the device stores in
bf16 (h, M_l(h), g, u, hf; dlogits, bf16(dx) before the FFN and the mixing
backward, the FFN pre-activation gradient, and the mixing's input gradient),
so that the device is compared with an fp64 computation that takes the same
roundings; the residual stream x and its gradient stay unrounded.
"""
from __future__ import annotations

import numpy as np

from . import oracle as O

EPS = 1e-5


def _rb(a, on):
    return O.round_bf16(a) if on else a


def ln_fwd(x, g, b):
    """LayerNorm over the last axis: (x - mean) / sqrt(var + eps) * g + b;
    returns (y, xhat, rstd)."""
    mu = x.mean(axis=-1, keepdims=True)
    xc = x - mu
    var = (xc * xc).mean(axis=-1, keepdims=True)
    rstd = 1.0 / np.sqrt(var + EPS)
    xhat = xc * rstd
    return xhat * g + b, xhat, rstd


def ln_bwd(dy, xhat, rstd, g):
    """Gradients of ln_fwd: (dx, dg, db) for upstream dy."""
    dxhat = dy * g
    d = xhat.shape[-1]
    dx = rstd * (dxhat - dxhat.sum(axis=-1, keepdims=True) / d
                 - xhat * (dxhat * xhat).sum(axis=-1, keepdims=True) / d)
    axes = tuple(range(dy.ndim - 1))
    return dx, (dy * xhat).sum(axis=axes), dy.sum(axis=axes)


def forward(pr, round_bf16=False):
    """Loss and the saved tensors of the block for the BlockProblem-like `pr`
    (float64 or exactly representable values)."""
    rb = round_bf16
    ids = np.asarray(pr.ids)
    B, n1 = ids.shape
    n = n1 - 1
    L = pr.W_self.shape[0]
    d = pr.E.shape[1]
    f64 = lambda a: np.asarray(a, dtype=np.float64)
    x = f64(pr.E)[ids[:, :n]] + f64(pr.P)[None]
    zero_bias = np.zeros(d)
    cache = {"layers": []}
    for l in range(L):
        c = {"x": x}
        h, c["xhat1"], c["rstd1"] = ln_fwd(x, f64(pr.ln1_g[l]), f64(pr.ln1_b[l]))
        h = _rb(h, rb)
        m = O.layer_fwd(h, pr.W_self[l], pr.W_nbr[l], zero_bias, l, -1, O.CAUSAL,
                        round_bf16=rb)
        x = x + m
        c["h"], c["xm"] = h, x
        g, c["xhat2"], c["rstd2"] = ln_fwd(x, f64(pr.ln2_g[l]), f64(pr.ln2_b[l]))
        g = _rb(g, rb)
        u = _rb(g @ f64(pr.W1[l]).T + f64(pr.b1[l]), rb)
        a = np.maximum(u, 0.0)
        x = x + a @ f64(pr.W2[l]).T + f64(pr.b2[l])
        c["g"], c["u"], c["a"] = g, u, a
        cache["layers"].append(c)
    hf, cache["xhatf"], cache["rstdf"] = ln_fwd(x, f64(pr.lnf_g), f64(pr.lnf_b))
    hf = _rb(hf, rb)
    logits = hf @ f64(pr.Wh).T + f64(pr.bh)
    mx = logits.max(axis=-1, keepdims=True)
    lse = mx[..., 0] + np.log(np.exp(logits - mx).sum(axis=-1))
    tgt = ids[:, 1:]
    picked = np.take_along_axis(logits, tgt[..., None], axis=-1)[..., 0]
    loss = float((lse - picked).mean())
    cache.update(hf=hf, logits=logits, lse=lse, xL=x)
    return loss, cache


def backward(pr, cache, round_bf16=False):
    """Gradients of the mean loss with respect to every parameter (a dict
    with the BlockProblem field names), by the chain rule through forward()."""
    rb = round_bf16
    ids = np.asarray(pr.ids)
    B, n1 = ids.shape
    n = n1 - 1
    L = pr.W_self.shape[0]
    V, d = pr.E.shape
    f64 = lambda a: np.asarray(a, dtype=np.float64)
    N = B * n
    # cross-entropy: d loss / d logits = (softmax - onehot) / N
    p = np.exp(cache["logits"] - cache["lse"][..., None])
    np.put_along_axis(p, ids[:, 1:, None], np.take_along_axis(p, ids[:, 1:, None], -1) - 1.0, -1)
    dlog = _rb(p / N, rb)
    hf = cache["hf"]
    gr = {"Wh": np.einsum("btv,btd->vd", dlog, hf), "bh": dlog.sum(axis=(0, 1))}
    dhf = dlog @ f64(pr.Wh)
    dx, gr["lnf_g"], gr["lnf_b"] = ln_bwd(dhf, cache["xhatf"], cache["rstdf"], f64(pr.lnf_g))
    names = ("ln1_g", "ln1_b", "W_self", "W_nbr", "ln2_g", "ln2_b", "W1", "b1", "W2", "b2")
    for k in names:
        gr[k] = np.zeros(np.shape(getattr(pr, k)))
    for l in reversed(range(L)):
        c = cache["layers"][l]
        # FFN sublayer: x_out = xm + relu(u) W2^T + b2, u = g W1^T + b1
        df = _rb(dx, rb)
        gr["W2"][l] = np.einsum("btd,bth->dh", df, c["a"])
        gr["b2"][l] = df.sum(axis=(0, 1))
        dpre = _rb((df @ f64(pr.W2[l])) * (c["u"] > 0), rb)
        gr["W1"][l] = np.einsum("bth,btd->hd", dpre, c["g"])
        gr["b1"][l] = dpre.sum(axis=(0, 1))
        dg = dpre @ f64(pr.W1[l])
        dxm, gr["ln2_g"][l], gr["ln2_b"][l] = ln_bwd(dg, c["xhat2"], c["rstd2"],
                                                     f64(pr.ln2_g[l]))
        dxm = dxm + dx
        # mixing sublayer: xm = x + M_l(h), h = LN1(x)
        dm = _rb(dxm, rb)
        dh, dWs, dWn, _ = O.layer_bwd(c["h"], c["h"], dm, pr.W_self[l], pr.W_nbr[l], l, -1,
                                      O.CAUSAL, round_bf16=rb)
        gr["W_self"][l], gr["W_nbr"][l] = dWs, dWn
        dx1, gr["ln1_g"][l], gr["ln1_b"][l] = ln_bwd(dh, c["xhat1"], c["rstd1"],
                                                     f64(pr.ln1_g[l]))
        dx = dx1 + dxm
    # x = E[ids] + P: rows of E gather the gradient of every position that reads them
    gE = np.zeros((V, d))
    np.add.at(gE, ids[:, :n].reshape(-1), dx.reshape(-1, d))
    gr["E"], gr["P"] = gE, dx.sum(axis=0)
    return gr


def relu_margins(pr, round_bf16=True):
    """Smallest |u| / std(u) over every FFN pre-activation u of the forward:
    how far the ReLU decisions sit from the kink."""
    _, cache = forward(pr, round_bf16=round_bf16)
    worst = np.inf
    for c in cache["layers"]:
        u = c["u"]
        worst = min(worst, float(np.abs(u).min() / max(u.std(), 1e-300)))
    return worst


def with_separated_relu_decisions(pr, round_bf16=True):
    """A copy of the block problem `pr` whose FFN biases b1 keep every ReLU
    decision of the forward clear of the kink (test-input construction, not
    part of the block).

    Two computations of the same forward (here fp64, on the device fp32)
    differ at rounding level, so a pre-activation within rounding of 0 can be
    switched on by one and off by the other; both answers are right, but an
    element-wise comparison of the gradients then fails on one token's row.
    Layer by layer, in forward order (b1 of layer l moves only what comes after
    it), this takes the pre-activations v = g W1^T of every hidden unit j over
    the B n tokens, finds the widest gap between neighbouring sorted values in
    their middle half, and sets b1[l, j] to minus the gap's midpoint (as an
    fp32 number): about half the tokens are active, the decisions still depend
    on the data, and each one sits half a gap (a few per cent of std(u) at
    these sizes) from 0."""
    import copy
    q = copy.copy(pr)
    b1 = np.array(pr.b1, dtype=np.float64).copy()
    L, h = b1.shape
    for l in range(L):
        q.b1 = b1.copy()
        _, cache = forward(q, round_bf16=round_bf16)
        v = (cache["layers"][l]["g"] @ np.asarray(pr.W1[l], dtype=np.float64).T).reshape(-1, h)
        N = v.shape[0]
        lo, hi = N // 4, max(N // 4 + 1, (3 * N) // 4)
        for j in range(h):
            s = np.sort(v[:, j])
            gaps = s[lo + 1:hi + 1] - s[lo:hi]
            k = lo + int(np.argmax(gaps))
            b1[l, j] = float(np.float32(-(s[k] + s[k + 1]) / 2))
    q.b1 = b1
    return q


def step(pr, round_bf16=False):
    """(loss, gradients) of one block step."""
    loss, cache = forward(pr, round_bf16=round_bf16)
    return loss, backward(pr, cache, round_bf16=round_bf16)
