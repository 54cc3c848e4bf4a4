"""Pins of the fp64 oracle against facts the paper and the mathematics fix.

None of these re-derives the oracle's own formula: each compares it with a
count the paper prints (tests/golden), a closed form, a structural fact found
by brute-force dependency propagation, an independent library routine
(numpy matmul, torch's bf16 conversion) or central finite differences.
"""
import json
import os

import numpy as np
import pytest

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _dims(spec, n, L):
    b = n.bit_length() - 1
    if spec == "rot":
        return [l % b for l in range(L)]
    if spec == "fixed0":
        return [0] * L
    return list(spec)


def _jacobian_structure(n, dims, causal, seed=0):
    """J[i, j] = d y_i / d x_j of a d = 1 linear stack, found by pushing the
    n basis vectors through the oracle (one per sample).  Random nonzero
    scalar weights make every structural path show up as a nonzero."""
    L = len(dims)
    r = np.random.default_rng(seed)
    Ws = r.uniform(0.5, 1.5, size=(L, 1, 1)) * r.choice([-1, 1], size=(L, 1, 1))
    Wn = r.uniform(0.5, 1.5, size=(L, 1, 1)) * r.choice([-1, 1], size=(L, 1, 1))
    x = np.eye(n).reshape(n, n, 1)            # sample j is the basis vector e_j
    y, _, _ = O.stack_fwd(x, Ws, Wn, None, 0, L, -1, O.CAUSAL if causal else 0, dims=dims)
    return y[:, :, 0].T                       # J[i, j]


# ---------------------------------------------------------------- partner rule

def test_partner_involution_and_single_bit():
    # partner of partner is self; partner differs in exactly bit s (Sec. 3.1)
    for b in range(1, 11):
        n = 1 << b
        for s in range(b):
            i = np.arange(n)
            p = np.array([O.partner(int(v), s) for v in i])
            q = np.array([O.partner(int(v), s) for v in p])
            assert np.array_equal(q, i)
            assert np.all(p != i)
            diff = p ^ i
            assert np.all(diff == (1 << s))


def test_partner_table_causal_keeps_earlier_endpoint():
    # causal rule: a position receives only from an earlier partner (Sec. 3.1)
    n = 64
    for layer in range(12):
        t = O.partner_table(layer, -1, n, O.CAUSAL)
        full = O.partner_table(layer, -1, n, 0)
        for i in range(n):
            assert full[i] >= 0
            if t[i] >= 0:
                assert t[i] == full[i] and t[i] < i
            else:
                assert full[i] > i
        assert (t >= 0).sum() == n // 2


def test_layer_dimension_rotates_and_fixed_control():
    assert [O.dim(l, -1, 64) for l in range(13)] == [0, 1, 2, 3, 4, 5, 0, 1, 2, 3, 4, 5, 0]
    assert [O.dim(l, 3, 64) for l in range(5)] == [3] * 5
    assert O.dim(0, 6, 64) == -1            # no such dimension
    assert O.dim(0, -1, 48) == -1           # n must be a power of two


# ---------------------------------------------------------------- link counts (paper tables)

@pytest.mark.parametrize("case", json.load(open(os.path.join(GOLDEN, "link_counts.json")))["cases"],
                         ids=lambda c: c["name"])
def test_link_counts_match_paper(case):
    n, L, causal = case["n"], case["L"], case["causal"]
    dims = _dims(case["dims"], n, L)
    total = 0
    for s in dims:
        J = _jacobian_structure(n, [s], causal)
        total += int(np.count_nonzero(np.abs(J) > 1e-12))
    assert total == case["links"], case["cite"]


def test_links_per_layer_closed_form():
    # per layer: 2n non-causal, 3n/2 causal (Table B1cost rot: 96 at n = 64)
    for n in (4, 16, 64, 256):
        b = n.bit_length() - 1
        for s in range(b):
            Jc = _jacobian_structure(n, [s], True)
            Jn = _jacobian_structure(n, [s], False)
            assert np.count_nonzero(Jc) == 3 * n // 2
            assert np.count_nonzero(Jn) == 2 * n


# ---------------------------------------------------------------- reach (brute force)

@pytest.mark.parametrize("case", json.load(open(os.path.join(GOLDEN, "reach.json")))["cases"],
                         ids=lambda c: c["name"])
def test_reach_claims(case):
    n, L = case["n"], case["L"]
    dims = _dims(case["dims"], n, L)
    J = np.abs(_jacobian_structure(n, dims, case["causal"])) > 1e-12
    i = np.arange(n)[:, None]
    j = np.arange(n)[None, :]
    exp = case["expect"]
    if exp == "all":
        assert J.all(), case["cite"]
    elif exp == "no_bit_5":
        across = ((i ^ j) & 32) != 0
        assert not J[across].any(), case["cite"]
        assert J[~across].all()
    elif exp == "exactly_2":
        assert (J.sum(axis=1) == 2).all(), case["cite"]
    elif exp == "submasks":
        sub = (j & ~i) == 0
        assert np.array_equal(J, sub), case["cite"]
        assert not J[j > i].any()       # causal: nothing from later positions
    else:
        raise AssertionError(exp)


def test_near_layer_links_one_predecessor():
    # Eq. (1) with k = 1 ("near", App. A): y_i depends on x_i and x_{i-1}, nothing else;
    # the first position of each sample has no predecessor: 2n - 1 links
    for n in (4, 16, 64, 256):
        J = np.abs(_jacobian_structure(n, [-1], True)) > 1e-12
        i = np.arange(n)[:, None]
        j = np.arange(n)[None, :]
        assert np.array_equal(J, (j == i) | (j == i - 1))
        assert J.sum() == 2 * n - 1
    # distance k: x_{i-k}, and the causal flag does not change a shift
    J = np.abs(_jacobian_structure(64, [-5], False)) > 1e-12
    i = np.arange(64)[:, None]
    j = np.arange(64)[None, :]
    assert np.array_equal(J, (j == i) | (j == i - 5))


def test_gray_order_visits():
    # Sec. 4: Gray order over 16 layers flips bit ctz(t): dim 0 eight times, dim 5 never
    dims = [((t & -t).bit_length() - 1) for t in range(1, 17)]
    assert dims == [0, 1, 0, 2, 0, 1, 0, 3, 0, 1, 0, 2, 0, 1, 0, 4]
    assert dims.count(0) == 8 and dims.count(5) == 0


# ---------------------------------------------------------------- closed forms

def _closed_form_identity(x, dims, a, c):
    """Non-causal stack with W_self = a I, W_nbr = c I and no bias/activation:
    y_i = sum_j prod_t f_t(i, j) x_j, where dimension t used m_t times gives
    f = ((a+c)^m + (a-c)^m)/2 if bit t of i and j agree, else ((a+c)^m - (a-c)^m)/2.
    (Each dimension acts as the 2x2 map [[a, c], [c, a]] on its bit; its m-th
    power has those entries.)"""
    B, n, d = x.shape
    b = n.bit_length() - 1
    m = [dims.count(t) for t in range(b)]
    y = np.zeros_like(x)
    for i in range(n):
        for j in range(n):
            f = 1.0
            for t in range(b):
                same = ((i >> t) & 1) == ((j >> t) & 1)
                p, q = (a + c) ** m[t], (a - c) ** m[t]
                f *= (p + q) / 2 if same else (p - q) / 2
            y[:, i, :] += f * x[:, j, :]
    return y


@pytest.mark.parametrize("dims,a,c", [([0, 1, 2, 3], 1.0, 1.0),
                                      ([0, 1, 2, 3, 0, 1], 0.7, -0.4),
                                      ([2, 2, 2], 0.3, 1.1),
                                      ([3, 1, 0, 2, 3], -0.5, 0.9)])
def test_identity_weight_closed_form(dims, a, c):
    n, d, B = 16, 3, 2
    x = np.random.default_rng(1).standard_normal((B, n, d))
    L = len(dims)
    Ws = np.stack([a * np.eye(d)] * L)
    Wn = np.stack([c * np.eye(d)] * L)
    y, _, _ = O.stack_fwd(x, Ws, Wn, None, 0, L, -1, 0, dims=dims)
    np.testing.assert_allclose(y, _closed_form_identity(x, dims, a, c), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("k,L,a,c", [(1, 5, 0.5, 1.5), (3, 4, -0.7, 0.9), (2, 7, 1.0, 1.0)])
def test_repeated_shift_closed_form(k, L, a, c):
    # L shift layers of distance k with W_self = a I, W_nbr = c I: the stack is
    # (a I + c S_k)^L with S_k the shift by k (zero past the sample start), so
    # y_i = sum_j C(L, j) a^(L-j) c^j x_{i - j k}  (binomial theorem; S_k^j = S_{jk})
    from math import comb
    n, d, B = 16, 3, 2
    x = np.random.default_rng(11).standard_normal((B, n, d))
    Ws = np.stack([a * np.eye(d)] * L)
    Wn = np.stack([c * np.eye(d)] * L)
    y, _, _ = O.stack_fwd(x, Ws, Wn, None, 0, L, -1, O.CAUSAL, dims=[-k] * L)
    ref = np.zeros_like(x)
    for i in range(n):
        for j in range(L + 1):
            if i - j * k >= 0:
                ref[:, i] += comb(L, j) * a ** (L - j) * c ** j * x[:, i - j * k]
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_shift_then_jump_by_hand():
    # near then jump 2 on n = 4, d = 1, W_self = 1, W_nbr = 1, non-causal jump:
    # after near: u = (x0, x0 + x1, x1 + x2, x2 + x3); the jump pairs i with i ^ 2
    x = np.array([1.0, 10.0, 100.0, 1000.0]).reshape(1, 4, 1)
    ones = np.ones((2, 1, 1))
    y, _, _ = O.stack_fwd(x, ones, ones, None, 0, 2, -1, 0, dims=[-1, 1])
    u = np.array([1.0, 11.0, 110.0, 1100.0])
    ref = np.array([u[0] + u[2], u[1] + u[3], u[2] + u[0], u[3] + u[1]])
    np.testing.assert_array_equal(y[0, :, 0], ref)


def test_sum_over_all_positions_after_b_layers():
    # invariant: identity weights, b rotated layers -> every output is the sum over all positions
    n, d, B = 32, 4, 3
    x = np.random.default_rng(2).standard_normal((B, n, d))
    L = 5
    I = np.stack([np.eye(d)] * L)
    y, _, _ = O.stack_fwd(x, I, I, None, 0, L, -1, 0)
    np.testing.assert_allclose(y, np.broadcast_to(x.sum(axis=1, keepdims=True), y.shape),
                               rtol=1e-12, atol=1e-12)


def test_causal_identity_is_subset_sum():
    # causal rule with identity maps over every dimension once: y_i = sum over submasks j of i
    # (the "parallel prefix scan" of Sec. 3.1, under the link-count reading)
    n, d, B = 32, 2, 2
    x = np.random.default_rng(3).standard_normal((B, n, d))
    L = 5
    I = np.stack([np.eye(d)] * L)
    y, _, _ = O.stack_fwd(x, I, I, None, 0, L, -1, O.CAUSAL)
    ref = np.zeros_like(x)
    for i in range(n):
        for j in range(n):
            if j & ~i == 0:
                ref[:, i] += x[:, j]
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("flags", [0, O.RESIDUAL, O.ACT_RELU, O.ACT_RELU | O.RESIDUAL | O.CAUSAL])
def test_zero_nbr_is_per_position_map(flags):
    # invariant: W_nbr = 0 reduces the layer to a per-position affine map (numpy matmul)
    B, n, d = 2, 8, 5
    r = np.random.default_rng(4)
    x = r.standard_normal((B, n, d))
    Ws = r.standard_normal((d, d))           # not symmetric: catches a transposed operand
    bias = r.standard_normal(d)
    y = O.layer_fwd(x, Ws, np.zeros((d, d)), bias, 1, -1, flags)
    z = x @ Ws.T + bias
    ref = np.maximum(z, 0) if flags & O.ACT_RELU else z
    if flags & O.RESIDUAL:
        ref = ref + x
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_nbr_only_twice_returns_home():
    # W_self = 0 and the same dimension twice: partner of partner is self, so
    # y = W2 W1 x_i per position (numpy matmul chain); non-symmetric W catch transposes
    B, n, d = 2, 16, 4
    r = np.random.default_rng(5)
    x = r.standard_normal((B, n, d))
    W1, W2 = r.standard_normal((d, d)), r.standard_normal((d, d))
    Z = np.zeros((2, d, d))
    y, _, _ = O.stack_fwd(x, Z, np.stack([W1, W2]), None, 0, 2, 2, 0)
    np.testing.assert_allclose(y, x @ W1.T @ W2.T, rtol=1e-12, atol=1e-12)


def test_self_map_orientation():
    # Eq. (1) applies W_self to the column vector x_i: y_o = sum_k W[o, k] x_k
    d = 3
    Ws = np.zeros((d, d))
    Ws[0, 2] = 1.0                            # y_0 picks x_2
    x = np.zeros((1, 2, d))
    x[0, 0, 2] = 5.0
    y = O.layer_fwd(x, Ws, np.zeros((d, d)), None, 0, -1, 0)
    assert y[0, 0, 0] == 5.0 and y[0, 0, 1] == 0.0 and y[0, 0, 2] == 0.0


# ---------------------------------------------------------------- backward

def _loss(x, Ws, Wn, bias, dims, flags, dy):
    y, _, _ = O.stack_fwd(x, Ws, Wn, bias, 0, len(dims), -1, flags, dims=dims)
    return float((y * dy).sum())


@pytest.mark.parametrize("flags,dims", [(0, [0, 2, 1]), (O.CAUSAL, [0, 2, 1]),
                                        (O.RESIDUAL | O.ACT_RELU, [0, 2, 1]),
                                        (O.CAUSAL | O.RESIDUAL | O.ACT_RELU, [0, 2, 1]),
                                        (O.CAUSAL | O.RESIDUAL | O.ACT_RELU, [-1, 2, -3]),
                                        (0, [-2, 0, -1])])
def test_backward_matches_central_differences(flags, dims):
    B, n, d = 2, 8, 3
    L = len(dims)
    # the first seed from 6 on whose pre-activations keep away from the ReLU kink
    # (central differences across it would not be a derivative)
    for seed in range(6, 40):
        r = np.random.default_rng(seed)
        x = r.standard_normal((B, n, d))
        Ws = r.standard_normal((L, d, d)) * 0.6
        Wn = r.standard_normal((L, d, d)) * 0.6
        bias = r.standard_normal((L, d)) * 0.3
        dy = r.standard_normal((B, n, d))
        y, acts, zs = O.stack_fwd(x, Ws, Wn, bias, 0, L, -1, flags, dims=dims)
        if not (flags & O.ACT_RELU) or np.abs(zs).min() > 1e-3:
            break
    else:
        raise AssertionError("no seed keeps the pre-activations off the ReLU kink")
    dx, dWs, dWn, db = O.stack_bwd(acts, zs, dy, Ws, Wn, 0, L, -1, flags, dims=dims)
    h = 1e-6

    def num_grad(arr, setter):
        g = np.zeros_like(arr)
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            p = arr.copy(); p[idx] += h
            m = arr.copy(); m[idx] -= h
            g[idx] = (setter(p) - setter(m)) / (2 * h)
        return g

    gx = num_grad(x, lambda v: _loss(v, Ws, Wn, bias, dims, flags, dy))
    gWs = num_grad(Ws, lambda v: _loss(x, v, Wn, bias, dims, flags, dy))
    gWn = num_grad(Wn, lambda v: _loss(x, Ws, v, bias, dims, flags, dy))
    gb = num_grad(bias, lambda v: _loss(x, Ws, Wn, v, dims, flags, dy))
    for got, ref in ((dx, gx), (dWs, gWs), (dWn, gWn), (db, gb)):
        np.testing.assert_allclose(got, ref, rtol=1e-6, atol=1e-6 * np.abs(ref).max())


@pytest.mark.parametrize("dims", [None, [-1, 3, -1, 2, -4, 0]])
def test_adjoint_identity_linear_stack(dims):
    # <dy, J v> = <J^T dy, v> for the linear (no bias, no activation) causal stack
    B, n, d = 2, 16, 4
    r = np.random.default_rng(7)
    L = 6
    Ws = r.standard_normal((L, d, d))
    Wn = r.standard_normal((L, d, d))
    v = r.standard_normal((B, n, d))
    dy = r.standard_normal((B, n, d))
    Jv, acts, zs = O.stack_fwd(v, Ws, Wn, None, 0, L, -1, O.CAUSAL, dims=dims)
    JTdy, _, _, _ = O.stack_bwd(acts, zs, dy, Ws, Wn, 0, L, -1, O.CAUSAL, dims=dims)
    lhs, rhs = float((dy * Jv).sum()), float((JTdy * v).sum())
    assert abs(lhs - rhs) <= 1e-10 * max(1.0, abs(lhs))


def test_layer_bwd_equals_stack_bwd_single_layer():
    B, n, d = 2, 8, 3
    r = np.random.default_rng(8)
    x = r.standard_normal((B, n, d))
    Ws, Wn = r.standard_normal((1, d, d)), r.standard_normal((1, d, d))
    bias = r.standard_normal((1, d))
    dy = r.standard_normal((B, n, d))
    flags = O.CAUSAL | O.RESIDUAL | O.ACT_RELU
    y, acts, zs = O.stack_fwd(x, Ws, Wn, bias, 3, 1, -1, flags)
    y1, z1 = O.layer_fwd(x, Ws[0], Wn[0], bias[0], 3, -1, flags, want_z=True)
    np.testing.assert_array_equal(y, y1)
    a = O.stack_bwd(acts, zs, dy, Ws, Wn, 3, 1, -1, flags)
    b = O.layer_bwd(x, z1, dy, Ws[0], Wn[0], 3, -1, flags)
    for u, v in zip(a, b):
        np.testing.assert_array_equal(np.asarray(u).reshape(np.asarray(v).shape), v)


# ---------------------------------------------------------------- bf16 rounding mode

def test_round_bf16_matches_torch_conversion():
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(9)
    vals = np.concatenate([
        r.standard_normal(4000).astype(np.float32),
        (r.standard_normal(1000) * 1e-38).astype(np.float32),     # subnormal range
        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8), 0.0, 2 ** -133,
                  3.3895313892515355e38], dtype=np.float32),       # ties and edges
    ])
    ref = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.round_bf16(vals.astype(np.float64))
    np.testing.assert_array_equal(got, ref)


def test_round_mode_stores_bf16_values():
    B, n, d = 2, 8, 16
    r = np.random.default_rng(10)
    x = O.round_bf16(r.standard_normal((B, n, d)))
    Ws = r.standard_normal((3, d, d)) * 0.25
    Wn = r.standard_normal((3, d, d)) * 0.25
    y, acts, zs = O.stack_fwd(x, Ws, Wn, None, 0, 3, -1, O.RESIDUAL | O.ACT_RELU, round_bf16=True)
    for a in (y, acts, zs):
        np.testing.assert_array_equal(a, O.round_bf16(a))
    y64, _, _ = O.stack_fwd(x, Ws, Wn, None, 0, 3, -1, O.RESIDUAL | O.ACT_RELU)
    assert np.abs(y - y64).max() <= 3 * 2 ** -8 * np.abs(y64).max()
