"""The seeded input recipes: reproducible draws with the distributions the
workloads state (N(0, 1) activations, N(0, std^2) weights and biases, Zipf(1.1)
byte ids, uniform ids over 16 symbols), the shapes of the workloads, and the
bf16 rounding both sides consume.  CPU only."""
import numpy as np
import pytest
import torch

from paper_2609_18145_gb300 import synth


def test_draws_are_reproducible_and_seed_dependent():
    a = synth.normal((4, 5), 7)
    assert np.array_equal(a, synth.normal((4, 5), 7))
    assert not np.array_equal(a, synth.normal((4, 5), 8))
    p, q = synth.problem(2, 16, 32, L=3, seed=5), synth.problem(2, 16, 32, L=3, seed=5)
    for f in ("x", "W_self", "W_nbr", "bias", "dy", "z"):
        assert np.array_equal(getattr(p, f), getattr(q, f)), f
    # every tensor of a problem comes from its own stream
    assert not np.array_equal(p.W_self, p.W_nbr)


def test_normal_moments():
    a = synth.normal((1 << 18,), 3, 0.25).astype(np.float64)
    assert abs(a.mean()) < 4 * 0.25 / 2 ** 9           # 4 standard errors
    assert abs(a.std() - 0.25) < 0.01 * 0.25
    assert a.dtype == np.float64 and synth.normal((2,), 1).dtype == np.float32


def test_problem_shapes_and_scales():
    B, n, d, L = 3, 16, 64, 4
    p = synth.problem(B, n, d, L=L, seed=1, w_std=0.05)
    assert p.x.shape == (B, n, d) and p.dy.shape == (B, n, d)
    assert p.W_self.shape == (L, d, d) and p.W_nbr.shape == (L, d, d)
    assert p.bias.shape == (L, d) and p.z.shape == (L, B, n, d)
    assert abs(p.W_self.std() - 0.05) < 0.005 and abs(p.bias.std() - 0.1) < 0.03
    # default weight scale N(0, 1/d)
    q = synth.problem(2, 16, 256, L=2, seed=2)
    assert abs(q.W_self.std() - (1 / 256) ** 0.5) < 0.002


def test_zipf_ids_follow_rank_power_law():
    ids = synth.zipf_ids(64, 4096, 11)
    assert ids.min() >= 0 and ids.max() < 256 and ids.dtype == np.int64
    counts = np.bincount(ids.ravel(), minlength=256).astype(np.float64)
    # byte r - 1 has probability proportional to r^-1.1
    r = np.arange(1, 257, dtype=np.float64)
    p = r ** -1.1 / (r ** -1.1).sum()
    total = counts.sum()
    for k in (0, 1, 2, 9, 99):
        expect = p[k] * total
        assert abs(counts[k] - expect) < 5 * np.sqrt(expect), k
    assert counts[0] / counts[1] == pytest.approx(2 ** 1.1, rel=0.02)


def test_uniform_ids_and_embedded_inputs():
    ids = synth.uniform_ids(256, 64, 3)
    assert ids.min() == 0 and ids.max() == 15
    counts = np.bincount(ids.ravel(), minlength=16)
    assert counts.min() > 0.9 * ids.size / 16 and counts.max() < 1.1 * ids.size / 16
    p = synth.problem(4, 64, 128, seed=9, x_ids="uniform16")
    # every position is one of the 16 rows of the embedding table
    rows = np.unique(p.x.reshape(-1, 128), axis=0)
    assert 1 <= len(rows) <= 16
    z = synth.problem(4, 64, 128, seed=9, x_ids="zipf256")
    assert len(np.unique(z.x.reshape(-1, 128), axis=0)) <= 256


def test_bf16_rounding_both_sides_consume():
    a = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5e-41, 3.3e38, 0.1],
                 dtype=np.float32)
    t, e = synth.to_bf16_exact(a)
    assert t.dtype == torch.bfloat16 and e.dtype == np.float64
    # the float64 copy holds exactly the bf16 values
    assert np.array_equal(e, t.to(torch.float32).numpy().astype(np.float64))
    # ties to even: 1 + 2^-8 is half way between 1 and 1 + 2^-7 (even: 1)
    assert e[1] == 1.0 and e[2] == 1.0 + 2 ** -6
    # every value has at most 8 significant bits
    m, _ = np.frexp(e[e != 0])
    assert np.all(m * 2 ** 8 == np.round(m * 2 ** 8))


@pytest.mark.parametrize("name,shape", [
    ("reach_n64_d128", (256, 64, 128, 6, False)),
    ("charlm_w64_d512", (64, 64, 512, 16, True)),
    ("charlm_w256_d512", (64, 256, 512, 16, True)),
    ("scale_n256_d1024", (4096, 256, 1024, 8, False)),
    ("scale_n4096_d1024", (256, 4096, 1024, 12, False)),
    ("scale_n65536_d1024", (16, 65536, 1024, 16, False)),
])
def test_workloads_have_the_stated_shapes(name, shape):
    w = synth.WORKLOADS[name]
    assert (w["B"], w["n"], w["d"], w["L"], w["causal"]) == shape
    if name.startswith("scale"):
        # 2^20 tokens a step and L = log2 n rotated layers
        assert w["B"] * w["n"] == 1 << 20 and w["L"] == int(np.log2(w["n"]))
