"""Pins of the fp64 oracle of the character-LM block (oracle/block.py), on the
CPU: finite differences, a closed form, causality, symbol-permutation
invariance and the LayerNorm moments."""
import copy

import numpy as np
import pytest

from oracle import block as OB
from paper_2609_18145_gb300 import synth

FIELDS = ("E", "P", "ln1_g", "ln1_b", "W_self", "W_nbr", "ln2_g", "ln2_b", "W1", "b1", "W2",
          "b2", "lnf_g", "lnf_b", "Wh", "bh")


def tiny(seed=3, B=2, n=8, d=8, h=16, V=7, L=2):
    pr = synth.block_problem(B, n, d, h, V, L, seed=seed)
    for f in FIELDS:
        setattr(pr, f, np.asarray(getattr(pr, f), dtype=np.float64))
    return pr


def test_gradients_match_central_differences():
    """Every parameter tensor: sampled entries of the analytic gradient equal
    (L(p + e) - L(p - e)) / 2e; a dropped term, sign or transposed operand
    anywhere in the backward fails this."""
    pr = tiny()
    loss, gr = OB.step(pr)
    rng = np.random.default_rng(5)
    eps = 1e-6
    for f in FIELDS:
        a = getattr(pr, f)
        for _ in range(4):
            idx = tuple(int(rng.integers(0, s)) for s in a.shape)
            keep = a[idx]
            a[idx] = keep + eps
            lp, _ = OB.forward(pr)
            a[idx] = keep - eps
            lm, _ = OB.forward(pr)
            a[idx] = keep
            fd = (lp - lm) / (2 * eps)
            an = gr[f][idx]
            assert abs(fd - an) <= 1e-6 + 1e-4 * abs(fd), (f, idx, fd, an)


def test_zero_head_gives_log_vocab_loss_and_bias_gradient_closed_form():
    """Wh = 0, bh = 0: every symbol has probability 1/V, so the loss is ln V and
    d loss / d bh_v = 1/V - (share of targets equal to v)."""
    pr = tiny()
    pr.Wh[:] = 0.0
    pr.bh[:] = 0.0
    loss, gr = OB.step(pr)
    V = pr.E.shape[0]
    assert loss == pytest.approx(np.log(V), rel=1e-12)
    tgt = np.asarray(pr.ids)[:, 1:].reshape(-1)
    share = np.bincount(tgt, minlength=V) / tgt.size
    np.testing.assert_allclose(gr["bh"], 1.0 / V - share, rtol=0, atol=1e-12)


def test_logits_before_a_changed_symbol_do_not_move():
    """Causal: changing the input symbol at position t0 changes no logit at any
    position t < t0 (through mixing, LayerNorm and FFN alike)."""
    pr = tiny()
    _, c0 = OB.forward(pr)
    t0 = 5
    pr2 = copy.deepcopy(pr)
    pr2.ids = np.array(pr.ids)
    pr2.ids[:, t0] = (pr2.ids[:, t0] + 1) % pr.E.shape[0]
    _, c1 = OB.forward(pr2)
    np.testing.assert_array_equal(c0["logits"][:, :t0], c1["logits"][:, :t0])
    assert not np.array_equal(c0["logits"][:, t0], c1["logits"][:, t0])


def test_loss_is_invariant_to_a_consistent_permutation_of_the_symbols():
    pr = tiny()
    loss, _ = OB.forward(pr)
    V = pr.E.shape[0]
    perm = np.random.default_rng(9).permutation(V)     # symbol v is renamed perm[v]
    inv = np.argsort(perm)
    pr2 = copy.deepcopy(pr)
    pr2.ids = perm[np.asarray(pr.ids)]
    pr2.E, pr2.Wh, pr2.bh = pr.E[inv], pr.Wh[inv], pr.bh[inv]
    loss2, _ = OB.forward(pr2)
    assert loss2 == pytest.approx(loss, rel=1e-12)


def test_layernorm_moments():
    x = np.random.default_rng(2).standard_normal((5, 3, 16)) * 3 + 1
    y, xhat, rstd = OB.ln_fwd(x, np.ones(16), np.zeros(16))
    np.testing.assert_allclose(y.mean(axis=-1), 0.0, atol=1e-12)
    var = x.var(axis=-1)
    np.testing.assert_allclose(y.var(axis=-1), var / (var + OB.EPS), rtol=1e-12)


def test_bf16_storage_mode_stays_close_to_fp64():
    pr = tiny()
    l64, g64 = OB.step(pr)
    l16, g16 = OB.step(pr, round_bf16=True)
    assert abs(l16 - l64) < 2e-2 * abs(l64)
    for f in FIELDS:
        scale = np.abs(g64[f]).max()
        assert np.abs(g16[f] - g64[f]).max() <= 5e-2 * scale + 1e-12, f


def test_separated_relu_decisions_change_only_b1_and_keep_a_margin():
    """The test-input construction behind the element-wise GPU parity: only
    the FFN biases move, every pre-activation ends up at least 1 % of its
    spread from the kink (it starts far closer), and the decisions still
    depend on the data (each hidden unit is on for some tokens and off for
    others)."""
    pr = synth.block_problem(2, 16, 64, 128, 11, 3, seed=7)
    q = OB.with_separated_relu_decisions(pr, round_bf16=True)
    for f in ("E", "P", "ln1_g", "ln1_b", "W_self", "W_nbr", "ln2_g", "ln2_b", "W1", "W2", "b2",
              "lnf_g", "lnf_b", "Wh", "bh"):
        assert np.array_equal(np.asarray(getattr(q, f)), np.asarray(getattr(pr, f))), f
    assert OB.relu_margins(pr) < 1e-3
    assert OB.relu_margins(q) >= 1e-2
    assert np.array_equal(np.asarray(q.b1, dtype=np.float32).astype(np.float64), q.b1)
    _, cache = OB.forward(q, round_bf16=True)
    for c in cache["layers"]:
        on = (c["u"] > 0).reshape(-1, c["u"].shape[-1]).mean(axis=0)
        assert on.min() > 0.1 and on.max() < 0.9
