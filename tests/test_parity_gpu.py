"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Tolerances (relative error = max|gpu - ref| / max|ref| per tensor):
  fp32 path 1e-5, bf16 path 2e-2 against the oracle's bf16-storage mode
  (the oracle rounds every stored activation to bf16, as the device does);
  partner tables bit-exact.
Inputs are the seeded generators of paper_2609_18145_gb300.synth; the bf16
cases hand the oracle the exact bf16 values the device sees.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_18145_gb300 import synth

pytestmark = pytest.mark.gpu

TOL_F32 = 1e-5
TOL_BF16 = 2e-2
CAUSAL, RESIDUAL, RELU = 1, 2, 4


@pytest.fixture(scope="module")
def H():
    from paper_2609_18145_gb300 import hcw
    hcw.lib()
    return hcw


def rel(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    assert np.isfinite(got).all()
    return float(np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30))


def dev(a, dtype):
    """numpy float32 -> (device tensor of dtype, float64 numpy of its exact values)."""
    if dtype == torch.bfloat16:
        t, a64 = synth.to_bf16_exact(a)
        return t.cuda(), a64
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.cuda(), t.double().numpy()


def host(t):
    return t.float().cpu().double().numpy()


def masks_from_z(z):
    """ReLU masks in the stack's format from pre-activations z [..., d]:
    int32 words [..., ceil(d/32)], bit o % 32 of word o // 32 = (z[..., o] > 0)."""
    z = np.asarray(z)
    d = z.shape[-1]
    wpr = (d + 31) // 32
    bits = np.zeros(z.shape[:-1] + (wpr * 32,), dtype=np.uint64)
    bits[..., :d] = z > 0
    words = (bits.reshape(z.shape[:-1] + (wpr, 32)) << np.arange(32, dtype=np.uint64)).sum(-1)
    return torch.from_numpy(words.astype(np.uint32).view(np.int32))


# ---------------------------------------------------------------- index code

@pytest.mark.parametrize("n", [2, 8, 64, 256, 65536])
@pytest.mark.parametrize("flags", [0, CAUSAL])
def test_device_partner_table_bit_exact(H, n, flags):
    b = n.bit_length() - 1
    for layer in range(2 * b + 1):
        got = H.hcw_partner_table_device(layer, n, flags).cpu().numpy()
        assert np.array_equal(got, O.partner_table(layer, -1, n, flags))
    got = H.hcw_partner_table_device(5, n, flags, dim_override=b - 1).cpu().numpy()
    assert np.array_equal(got, O.partner_table(5, b - 1, n, flags))


# ---------------------------------------------------------------- single layer

LAYER_CASES_F32 = [
    # B, n, d, layer, dim_override
    (4, 16, 32, 0, -1), (4, 16, 32, 3, -1), (3, 8, 20, 2, -1), (2, 64, 96, 5, -1),
    (1, 2, 33, 0, -1), (4, 16, 32, 9, 1),
]
LAYER_CASES_BF16 = [
    (8, 16, 64, 0, -1),       # k = 1, one ragged row block
    (3, 16, 64, 2, -1),       # 24 rows per bit value (ragged)
    (2, 2, 64, 0, -1),        # n = 2, a single position per bit value and sample
    (16, 64, 128, 5, -1),     # k = 32
    (4, 256, 512, 7, -1),     # k = 128 (the 128-row box along lo)
    (4, 256, 512, 3, -1),     # k = 8
    (2, 64, 192, 4, -1),      # d = 192: 64-wide column tiles, ragged 128-row o tiles in dW
    (1, 4096, 64, 11, -1),    # k = 2048 > 128
    (5, 32, 256, 1, 0),       # fixed-dimension control, odd B
]
FLAG_SETS = [0, CAUSAL, CAUSAL | RESIDUAL, RESIDUAL | RELU, CAUSAL | RESIDUAL | RELU]


@pytest.mark.parametrize("flags", FLAG_SETS)
@pytest.mark.parametrize("case", LAYER_CASES_F32 + LAYER_CASES_BF16)
def test_layer_forward(H, case, flags):
    B, n, d, layer, dim = case
    dtype = torch.float32 if case in LAYER_CASES_F32 else torch.bfloat16
    pr = synth.problem(B, n, d, L=1, seed=B * 1000 + n + d + layer)
    x, x64 = dev(pr.x, dtype)
    Ws, Ws64 = dev(pr.W_self[0], dtype)
    Wn, Wn64 = dev(pr.W_nbr[0], dtype)
    bias = torch.from_numpy(pr.bias[0]).cuda()
    y, z = H.hcw_layer_fwd(x, Ws, Wn, bias, layer, dim, flags, want_z=True)
    torch.cuda.synchronize()
    rb = dtype == torch.bfloat16
    yr, zr = O.layer_fwd(x64, Ws64, Wn64, pr.bias[0].astype(np.float64), layer, dim, flags,
                         round_bf16=rb, want_z=True)
    tol = TOL_BF16 if rb else TOL_F32
    assert rel(host(y), yr) <= tol
    assert rel(host(z), zr) <= tol


@pytest.mark.parametrize("flags", FLAG_SETS)
@pytest.mark.parametrize("case", LAYER_CASES_F32 + LAYER_CASES_BF16)
def test_layer_backward(H, case, flags):
    B, n, d, layer, dim = case
    dtype = torch.float32 if case in LAYER_CASES_F32 else torch.bfloat16
    pr = synth.problem(B, n, d, L=1, seed=B * 1000 + n + d + layer + 7)
    x, x64 = dev(pr.x, dtype)
    z, z64 = dev(pr.z[0], dtype)            # a given pre-activation: same ReLU mask on both sides
    dy, dy64 = dev(pr.dy, dtype)
    Ws, Ws64 = dev(pr.W_self[0], dtype)
    Wn, Wn64 = dev(pr.W_nbr[0], dtype)
    dx, gWs, gWn, gb = H.hcw_layer_bwd(x, z, dy, Ws, Wn, layer, dim, flags)
    torch.cuda.synchronize()
    rb = dtype == torch.bfloat16
    rdx, rWs, rWn, rb_ = O.layer_bwd(x64, z64, dy64, Ws64, Wn64, layer, dim, flags,
                                     round_bf16=rb)
    tol = TOL_BF16 if rb else TOL_F32
    assert rel(host(dx), rdx) <= tol
    assert rel(host(gWs), rWs) <= (1e-5 if not rb else 1e-4)
    assert rel(host(gWn), rWn) <= (1e-5 if not rb else 1e-4)
    assert rel(host(gb), rb_) <= (1e-5 if not rb else 1e-4)


@pytest.mark.parametrize("flags", [CAUSAL | RESIDUAL | RELU, RESIDUAL])
def test_many_tiles_per_cta(H, flags):
    """B = 256 sequences of n = 256 at d = 512 give 1024 forward / input-gradient
    tiles, several per persistent CTA: every TMEM accumulator is reused, which
    the smaller cases never do.  Checked on sampled sequences against the oracle."""
    B, n, d, layer = 256, 256, 512, 6
    pr = synth.problem(B, n, d, L=1, seed=21, w_std=(1 / (2 * d)) ** 0.5)
    x, x64 = dev(pr.x, torch.bfloat16)
    Ws, Ws64 = dev(pr.W_self[0], torch.bfloat16)
    Wn, Wn64 = dev(pr.W_nbr[0], torch.bfloat16)
    dy, dy64 = dev(pr.dy, torch.bfloat16)
    z, z64 = dev(pr.z[0], torch.bfloat16)
    bias = torch.from_numpy(pr.bias[0]).cuda()
    y, zs = H.hcw_layer_fwd(x, Ws, Wn, bias, layer, -1, flags, want_z=True)
    dx = H.hcw_layer_bwd_data(dy, dy, Ws, Wn, layer, -1, flags)
    assert H.hcw_sync_status() == H.HCW_OK
    picks = [0, 77, 128, 255]
    yr, zr = O.layer_fwd(x64[picks], Ws64, Wn64, pr.bias[0].astype(np.float64), layer, -1, flags,
                         round_bf16=True, want_z=True)
    assert rel(host(y)[picks], yr) <= TOL_BF16
    assert rel(host(zs)[picks], zr) <= TOL_BF16
    rdx, _, _, _ = O.layer_bwd(x64[picks], z64[picks], dy64[picks], Ws64, Wn64, layer, -1,
                               flags & ~RELU, round_bf16=True)
    assert rel(host(dx)[picks], rdx) <= TOL_BF16


def test_backward_is_deterministic(H):
    pr = synth.problem(8, 256, 512, L=1, seed=3)
    x, _ = dev(pr.x, torch.bfloat16)
    dy, _ = dev(pr.dy, torch.bfloat16)
    Ws, _ = dev(pr.W_self[0], torch.bfloat16)
    Wn, _ = dev(pr.W_nbr[0], torch.bfloat16)
    a = H.hcw_layer_bwd(x, None, dy, Ws, Wn, 4, -1, CAUSAL | RESIDUAL)
    b = H.hcw_layer_bwd(x, None, dy, Ws, Wn, 4, -1, CAUSAL | RESIDUAL)
    for u, v in zip(a, b):
        assert torch.equal(u, v)


def test_empty_batch(H):
    x = torch.empty(0, 16, 64, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(64, 64, dtype=torch.bfloat16, device="cuda")
    y = H.hcw_layer_fwd(x, W, W, None, 0)
    assert y.shape == x.shape
    dx, gWs, gWn, gb = H.hcw_layer_bwd(x, None, x, W, W, 0)
    torch.cuda.synchronize()
    assert float(gWs.abs().sum()) == 0.0 and float(gWn.abs().sum()) == 0.0
    assert float(gb.abs().sum()) == 0.0


# ---------------------------------------------------------------- stacks

def run_stack(H, pr, dtype, L, flags, layer0=0, dim=-1):
    """Forward: device stack vs oracle stack on the same inputs.  Backward: the
    device stack backward is fed the oracle's saved layer inputs and
    pre-activations (bf16-exact in bf16 mode), so that both sides take the
    same ReLU decisions; near-zero pre-activations would otherwise be decided
    differently by two forwards that differ by rounding, and both answers are
    valid.  Returns (device, oracle) tuples (y, acts, dx, dW_self, dW_nbr, dbias)."""
    x, x64 = dev(pr.x, dtype)
    Ws, Ws64 = dev(pr.W_self, dtype)
    Wn, Wn64 = dev(pr.W_nbr, dtype)
    bias = torch.from_numpy(pr.bias).cuda()
    dy, dy64 = dev(pr.dy, dtype)
    y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, layer0, dim, flags)
    rb = dtype == torch.bfloat16
    ry, racts, rzs = O.stack_fwd(x64, Ws64, Wn64, pr.bias.astype(np.float64), layer0, L, dim,
                                 flags, round_bf16=rb)
    o_acts = torch.from_numpy(racts[1:]).to(dtype).cuda() if L > 1 else None
    o_masks = masks_from_z(rzs).cuda() if flags & RELU else None
    dx, gWs, gWn, gb = H.hcw_stack_bwd(x, o_acts, o_masks, dy, Ws, Wn, layer0, dim, flags)
    torch.cuda.synchronize()
    rdx, rWs, rWn, rgb = O.stack_bwd(racts, rzs, dy64, Ws64, Wn64, layer0, L, dim, flags,
                                     round_bf16=rb)
    dev_acts = host(acts) if L > 1 else np.zeros((0,) + pr.x.shape)
    return ((host(y), dev_acts, host(dx), host(gWs), host(gWn), host(gb)),
            (ry, racts[1:], rdx, rWs, rWn, rgb))


WHAT = ("y", "acts", "dx", "dW_self", "dW_nbr", "dbias")


STACK_CASES = [
    # name, dtype, B, n, d, L, flags, w_std
    ("tiny_n16_d32_f32", torch.float32, 4, 16, 32, 4, 0, None),
    ("tiny_n16_d32_f32_causal_res_relu", torch.float32, 4, 16, 32, 4,
     CAUSAL | RESIDUAL | RELU, None),
    ("tiny_n16_d64_bf16", torch.bfloat16, 4, 16, 64, 4, 0, None),
    ("n16_d64_bf16_8layers_causal_res", torch.bfloat16, 6, 16, 64, 8, CAUSAL | RESIDUAL,
     (1 / 128) ** 0.5),
    ("n64_d128_bf16_causal_res_relu", torch.bfloat16, 8, 64, 128, 6, CAUSAL | RESIDUAL | RELU,
     (1 / 256) ** 0.5),
    ("n256_d512_bf16_causal_res_relu", torch.bfloat16, 2, 256, 512, 16,
     CAUSAL | RESIDUAL | RELU, (1 / 1024) ** 0.5),
    # 256-column tiles on pairs of SMs with an odd number of 128-row blocks (the
    # last pair's second CTA has no rows)
    ("n64_d256_bf16_odd_row_blocks", torch.bfloat16, 10, 64, 256, 6,
     CAUSAL | RESIDUAL | RELU, (1 / 512) ** 0.5),
    ("n64_d256_bf16_odd_row_blocks_noncausal", torch.bfloat16, 10, 64, 256, 6,
     RESIDUAL, (1 / 512) ** 0.5),
    # d = 192: 64-column tiles and a ragged 128-row o tile in the weight
    # gradient, whose few tiles take the launch over token splits of every layer
    ("n64_d192_bf16_split_weight_gradient", torch.bfloat16, 4, 64, 192, 5,
     CAUSAL | RESIDUAL | RELU, (1 / 384) ** 0.5),
]


@pytest.mark.parametrize("case", STACK_CASES, ids=lambda c: c[0])
def test_stack_forward_backward(H, case):
    name, dtype, B, n, d, L, flags, w_std = case
    pr = synth.problem(B, n, d, L=L, seed=11, w_std=w_std)
    got, ref = run_stack(H, pr, dtype, L, flags)
    tol = TOL_BF16 if dtype == torch.bfloat16 else TOL_F32
    for g, r, what in zip(got, ref, WHAT):
        if g.size:
            assert rel(g, r) <= tol, (name, what, rel(g, r))


@pytest.fixture
def resident(H):
    """Run the bf16 stacks on the resident kernels wherever the shape fits."""
    prev = H.hcw_set_stack_kernels(H.HCW_STACK_RESIDENT)
    yield
    H.hcw_set_stack_kernels(prev)


RESIDENT_CASES = [
    # name, B, n, d, L, flags, w_std, layer0, dim: every shape fits the resident
    # kernels (d in {128, 256, 512}, n <= 256, B*n a multiple of 256)
    # n = 256: the layers with s = 7 use the other CTA split (rows change CTA twice
    # per rotation); two accumulator chunks of 256 columns
    ("n256_d512_causal_res_relu", 2, 256, 512, 16, CAUSAL | RESIDUAL | RELU, (1 / 1024) ** 0.5,
     0, -1),
    # both partner windows, starting mid-rotation
    ("n256_d512_noncausal_res", 2, 256, 512, 10, RESIDUAL, (1 / 1024) ** 0.5, 3, -1),
    # chunks of 128 columns; no residual (the input gradient starts each layer from 0)
    ("n256_d256_causal_relu", 2, 256, 256, 9, CAUSAL | RELU, (1 / 512) ** 0.5, 5, -1),
    # two samples of 128 per CTA pair, no split change
    ("n128_d512_causal_res", 2, 128, 512, 7, CAUSAL | RESIDUAL, (1 / 1024) ** 0.5, 0, -1),
    # one accumulator chunk (d = 128), eight samples of 32 per pair
    ("n32_d128_noncausal_relu", 8, 32, 128, 5, RELU, (1 / 256) ** 0.5, 0, -1),
    # the fixed control on dimension 7: every layer on the other split
    ("n256_d128_dim7", 2, 256, 128, 4, CAUSAL | RESIDUAL | RELU, (1 / 256) ** 0.5, 0, 7),
    # 20 layers: two launches, the second continuing from the first's output
    # (forward) and from its fp32 residual stream (input gradient)
    ("n256_d128_20_layers", 2, 256, 128, 20, CAUSAL | RESIDUAL | RELU, (1 / 256) ** 0.5, 0, -1),
]


@pytest.mark.parametrize("case", RESIDENT_CASES, ids=lambda c: c[0])
def test_resident_stack_forward_backward(H, resident, case):
    name, B, n, d, L, flags, w_std, layer0, dim = case
    pr = synth.problem(B, n, d, L=L, seed=13, w_std=w_std)
    got, ref = run_stack(H, pr, torch.bfloat16, L, flags, layer0=layer0, dim=dim)
    assert H.hcw_sync_status() == H.HCW_OK
    for g, r, what in zip(got, ref, WHAT):
        if g.size:
            assert rel(g, r) <= TOL_BF16, (name, what, rel(g, r))


@pytest.mark.parametrize("flags", [CAUSAL | RESIDUAL | RELU, RESIDUAL, CAUSAL])
def test_resident_and_streaming_stacks_agree(H, flags):
    """The same stack on both kernel families.  Forward: the resident kernel
    sums the self and partner products K block by K block (the streaming one
    sums the self part first), so y and the saved activations agree to bf16
    rounding and only pre-activations within rounding of 0 may take the other
    ReLU decision.  Input gradient: the resident kernel keeps the residual
    stream in fp32 between layers (the streaming one rounds it to bf16 at
    each), so dx and the weight gradients agree to bf16 rounding."""
    B, n, d, L = 4, 256, 512, 9
    pr = synth.problem(B, n, d, L=L, seed=17, w_std=(1 / (2 * d)) ** 0.5)
    x, _ = dev(pr.x, torch.bfloat16)
    Ws, _ = dev(pr.W_self, torch.bfloat16)
    Wn, _ = dev(pr.W_nbr, torch.bfloat16)
    dy, _ = dev(pr.dy, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    out = {}
    saved = None
    for mode in (H.HCW_STACK_STREAMING, H.HCW_STACK_RESIDENT):
        prev = H.hcw_set_stack_kernels(mode)
        try:
            y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, 2, -1, flags)
            # both backwards run on the streaming forward's saved state (same ReLU
            # decisions)
            saved = saved or (acts, masks)
            res = H.hcw_stack_bwd(x, saved[0], saved[1], dy, Ws, Wn, 2, -1, flags)
            torch.cuda.synchronize()
            assert H.hcw_sync_status() == H.HCW_OK
        finally:
            H.hcw_set_stack_kernels(prev)
        out[mode] = (y, acts, masks) + tuple(res)
    a, b = out[H.HCW_STACK_STREAMING], out[H.HCW_STACK_RESIDENT]
    assert rel(host(b[0]), host(a[0])) <= 1e-2 and rel(host(b[1]), host(a[1])) <= 1e-2
    if flags & RELU:
        differ = torch.bitwise_xor(a[2], b[2])
        flipped = int(sum(bin(int(w) & 0xFFFFFFFF).count("1") for w in differ.flatten().cpu()
                          if int(w) != 0))
        assert flipped <= 1e-3 * a[2].numel() * 32, flipped
    for i, what in ((3, "dx"), (4, "dW_self"), (5, "dW_nbr"), (6, "dbias")):
        assert rel(host(b[i]), host(a[i])) <= 1e-2, what


def gray_dims(L):
    """Dimension flipped at each step of the binary reflected Gray code (Sec. 4: it
    visits dimension 0 every other layer and dimension b-1 only late)."""
    return [(g & -g).bit_length() - 1 for g in range(1, L + 1)]


SCHEDULE_CASES = [
    # name, kernels, B, n, d, flags, dims
    ("gray16_n64", "auto", 8, 64, 128, CAUSAL | RESIDUAL | RELU, gray_dims(16)),
    ("perm_twice_n64", "auto", 8, 64, 128, RESIDUAL, [3, 0, 5, 1, 4, 2, 2, 4, 1, 5, 0, 3]),
    ("gray16_n64_resident", "resident", 8, 64, 128, CAUSAL | RESIDUAL | RELU, gray_dims(16)),
    # n = 256: dimension 7 at irregular places (twice in a row, first, last):
    # the resident kernels change CTA split there
    ("n256_dim7_resident", "resident", 2, 256, 128, CAUSAL | RESIDUAL | RELU,
     [7, 7, 0, 3, 7, 6, 5, 7]),
    ("n256_dim7_streaming", "streaming", 2, 256, 128, CAUSAL | RESIDUAL | RELU,
     [7, 7, 0, 3, 7, 6, 5, 7]),
    # shift layers of Eq. (1) (-k; near = -1): the mixa schedule at window 64
    # (Sec. 3.3: local and long-range layers alternate, jumps 32 .. 1)
    ("mixa_n64", "auto", 8, 64, 128, CAUSAL | RESIDUAL | RELU,
     [-1, 5, -1, 4, -1, 3, -1, 2, -1, 1, -1, 0]),
    # the near and jump layers of the hybrid256 schedule (App. A, attention left out)
    ("hybrid256_sparse_n256", "auto", 2, 256, 128, CAUSAL | RESIDUAL | RELU,
     [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0]),
    # long shifts, no activation, d = 256 tiles
    ("long_shifts_n128_d256", "auto", 4, 128, 256, RESIDUAL, [-3, -64, 2, -127, -1]),
    # enough layers and tiles at d = 512 for the batched weight-gradient launch
    # on SM pairs, shift layers included (their partner rows read at p - k)
    ("hybrid256_n256_d512_batched_dw", "auto", 2, 256, 512, CAUSAL | RESIDUAL | RELU,
     [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0]),
    ("long_shifts_n256_d512_batched_dw", "auto", 2, 256, 512, RESIDUAL,
     [-3, -64, 2, -127, -1, 5, -200, 0, -1, 7, -2, 3, -130, -255]),
    # n = 128 with an odd batch: the tokens are not whole 256-token row-block
    # pairs, so shift schedules run layer by layer
    ("shifts_n128_b3_layer_by_layer", "auto", 3, 128, 128, CAUSAL | RESIDUAL | RELU,
     [-1, 6, -2, 3, -127, 0]),
    # 20 layers: two stacked launches, shifts on both sides of the boundary
    ("mixed20_n256_d256", "auto", 2, 256, 256, CAUSAL | RESIDUAL | RELU,
     [-1, 7, -3, 6, -1, 5, -100, 4, -1, 3, -255, 2, -1, 1, -17, 0, -1, 7, -2, 6]),
]


@pytest.mark.parametrize("case", SCHEDULE_CASES, ids=lambda c: c[0])
def test_stack_with_a_schedule_array(H, case):
    """hcw_stack_fwd_dims / hcw_stack_bwd_dims against the oracle's stacks on
    the same schedule (Sec. 3.3 schedules; Sec. 4 permutation and Gray order)."""
    name, kernels, B, n, d, flags, dims = case
    L = len(dims)
    pr = synth.problem(B, n, d, L=L, seed=19, w_std=(1 / (2 * d)) ** 0.5)
    mode = {"auto": H.HCW_STACK_AUTO, "resident": H.HCW_STACK_RESIDENT,
            "streaming": H.HCW_STACK_STREAMING}[kernels]
    prev = H.hcw_set_stack_kernels(mode)
    try:
        x, x64 = dev(pr.x, torch.bfloat16)
        Ws, Ws64 = dev(pr.W_self, torch.bfloat16)
        Wn, Wn64 = dev(pr.W_nbr, torch.bfloat16)
        dy, dy64 = dev(pr.dy, torch.bfloat16)
        bias = torch.from_numpy(pr.bias).cuda()
        y, acts, masks = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
        ry, racts, rzs = O.stack_fwd(x64, Ws64, Wn64, pr.bias.astype(np.float64), 0, L, -1,
                                     flags, round_bf16=True, dims=dims)
        assert rel(host(y), ry) <= TOL_BF16, name
        assert rel(host(acts), racts[1:]) <= TOL_BF16, name
        o_acts = torch.from_numpy(racts[1:]).to(torch.bfloat16).cuda()
        o_masks = masks_from_z(rzs).cuda() if flags & RELU else None
        dx, gWs, gWn, gb = H.hcw_stack_bwd_dims(x, o_acts, o_masks, dy, Ws, Wn, dims, flags)
        torch.cuda.synchronize()
        assert H.hcw_sync_status() == H.HCW_OK
        rdx, rWs, rWn, rgb = O.stack_bwd(racts, rzs, dy64, Ws64, Wn64, 0, L, -1, flags,
                                         round_bf16=True, dims=dims)
        for got, ref, what in ((dx, rdx, "dx"), (gWs, rWs, "dW_self"), (gWn, rWn, "dW_nbr"),
                               (gb, rgb, "dbias")):
            assert rel(host(got), ref) <= TOL_BF16, (name, what)
    finally:
        H.hcw_set_stack_kernels(prev)


@pytest.mark.parametrize("flags", [CAUSAL | RESIDUAL | RELU, 0])
def test_shift_schedule_fp32(H, flags):
    """The fp32 path (CUDA-core kernels) on a schedule of near, jump and shift
    layers against the oracle at the fp32 tolerance."""
    B, n, d = 3, 32, 48
    dims = [-1, 4, -1, 3, -5, 0, -1]
    L = len(dims)
    pr = synth.problem(B, n, d, L=L, seed=29, w_std=(1 / (2 * d)) ** 0.5)
    x, x64 = dev(pr.x, torch.float32)
    Ws, Ws64 = dev(pr.W_self, torch.float32)
    Wn, Wn64 = dev(pr.W_nbr, torch.float32)
    dy, dy64 = dev(pr.dy, torch.float32)
    bias = torch.from_numpy(pr.bias).cuda()
    y, acts, masks = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
    ry, racts, rzs = O.stack_fwd(x64, Ws64, Wn64, pr.bias.astype(np.float64), 0, L, -1, flags,
                                 dims=dims)
    assert rel(host(y), ry) <= TOL_F32 and rel(host(acts), racts[1:]) <= TOL_F32
    o_acts = torch.from_numpy(racts[1:]).float().cuda()
    o_masks = masks_from_z(rzs).cuda() if flags & RELU else None
    dx, gWs, gWn, gb = H.hcw_stack_bwd_dims(x, o_acts, o_masks, dy, Ws, Wn, dims, flags)
    torch.cuda.synchronize()
    rdx, rWs, rWn, rgb = O.stack_bwd(racts, rzs, dy64, Ws64, Wn64, 0, L, -1, flags, dims=dims)
    for got, ref, what in ((dx, rdx, "dx"), (gWs, rWs, "dW_self"), (gWn, rWn, "dW_nbr"),
                           (gb, rgb, "dbias")):
        assert rel(host(got), ref) <= TOL_F32, what


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_schedule_array_of_the_rotation_equals_the_rotated_stack(H, dtype):
    """dims = (layer0 + l) mod log2 n reproduces hcw_stack_fwd / hcw_stack_bwd
    with that layer0 exactly (the same kernels run on the same dimensions)."""
    B, n, d, L, layer0 = 4, 64, 64 if dtype == torch.float32 else 128, 9, 2
    flags = CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=23, w_std=(1 / (2 * d)) ** 0.5)
    x, _ = dev(pr.x, dtype)
    Ws, _ = dev(pr.W_self, dtype)
    Wn, _ = dev(pr.W_nbr, dtype)
    dy, _ = dev(pr.dy, dtype)
    bias = torch.from_numpy(pr.bias).cuda()
    dims = [(layer0 + l) % 6 for l in range(L)]
    a = H.hcw_stack_fwd(x, Ws, Wn, bias, layer0, -1, flags)
    b = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
    for u, v in zip(a, b):
        assert torch.equal(u, v)
    ga = H.hcw_stack_bwd(x, a[1], a[2], dy, Ws, Wn, layer0, -1, flags)
    gb = H.hcw_stack_bwd_dims(x, a[1], a[2], dy, Ws, Wn, dims, flags)
    for u, v in zip(ga, gb):
        assert torch.equal(u, v)


DECODE_CASES = [
    # name, B, n, d, flags, dims (None = rot), layer0, L
    ("rot_n64", 4, 64, 128, CAUSAL | RESIDUAL | RELU, None, 0, 12),
    ("rot_n64_from_layer3_no_relu", 3, 64, 64, CAUSAL | RESIDUAL, None, 3, 7),
    ("mixa_n64", 4, 64, 128, CAUSAL | RESIDUAL | RELU, [-1, 5, -1, 4, -1, 3, -1, 2, -1, 1, -1, 0],
     0, 12),
    ("hybrid256_sparse_n256", 2, 256, 128, CAUSAL | RESIDUAL | RELU,
     [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0], 0, 14),
    # two row blocks (the second ragged), a cluster of 10 CTAs of 64 columns,
    # weight chunks 128 wide
    ("rot_n32_B20_d640", 20, 32, 640, CAUSAL | RESIDUAL | RELU, None, 1, 5),
    # d = 1024: 16 CTAs of 64 columns, 8 chunks a part; d = 192: 12 CTAs of 16
    ("rot_n16_B3_d1024", 3, 16, 1024, CAUSAL | RESIDUAL | RELU, None, 0, 4),
    ("mixa_n32_B33_d192", 33, 32, 192, CAUSAL | RESIDUAL | RELU, [-1, 4, -3, 2, 1, -1, 0], 0, 7),
    # one sequence, one layer, d = 64 (a cluster of 4); 17 sequences at d = 256
    # (16 CTAs of 16 columns, a ragged second row block), no residual
    ("rot_n8_B1_d64_L1", 1, 8, 64, CAUSAL | RESIDUAL | RELU, None, 2, 1),
    ("rot_n16_B17_d256_plain", 17, 16, 256, CAUSAL | RELU, None, 0, 3),
]


@pytest.fixture(params=["warp_mma", "tcgen05"])
def decode_kernel(H, request):
    """Run the test under each contraction of hcw_decode_step."""
    mode = H.HCW_DECODE_WARP_MMA if request.param == "warp_mma" else H.HCW_DECODE_TCGEN05
    prev = H.hcw_set_decode_kernel(mode)
    yield request.param
    H.hcw_set_decode_kernel(prev)


@pytest.mark.parametrize("case", DECODE_CASES, ids=lambda c: c[0])
def test_decode_steps_reproduce_the_window_forward(H, case, decode_kernel):
    """Sec. 6: decoding one token at a time with bounded rings gives, at every
    position t, the output row t of the stack run over the whole window: the
    oracle's forward (bf16 storage) at the bf16 tolerance, and the device's
    stacked forward likewise."""
    name, B, n, d, flags, dims, layer0, L = case
    pr = synth.problem(B, n, d, L=L, seed=31, w_std=(1 / (2 * d)) ** 0.5)
    x, x64 = dev(pr.x, torch.bfloat16)
    Ws, Ws64 = dev(pr.W_self, torch.bfloat16)
    Wn, Wn64 = dev(pr.W_nbr, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    cache = torch.empty(H.hcw_decode_cache_bytes(L, B, n, d, dims=dims, layer0=layer0),
                        dtype=torch.uint8, device="cuda")
    ys = torch.empty_like(x)
    for t in range(n):
        xt = x[:, t].contiguous()
        ys[:, t] = H.hcw_decode_step(xt, Ws, Wn, bias, t, n, cache, flags, dims=dims,
                                     layer0=layer0)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    ry, _, _ = O.stack_fwd(x64, Ws64, Wn64, pr.bias.astype(np.float64), layer0, L, -1, flags,
                           round_bf16=True, dims=dims)
    assert rel(host(ys), ry) <= TOL_BF16, name
    if dims is None:
        y, _, _ = H.hcw_stack_fwd(x, Ws, Wn, bias, layer0, -1, flags)
    else:
        y, _, _ = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
    assert rel(host(ys), host(y)) <= TOL_BF16, name


def test_decode_full_size_window(H, decode_kernel):
    """The decode shape bench.py times (64 sequences, window 256, d = 512, 16
    rotated causal layers): every position of every sequence equals the
    device's stack forward over the window, and the first two sequences equal
    the oracle's window forward (bf16 storage)."""
    B, n, d, L = 64, 256, 512, 16
    flags = CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=41, w_std=(1 / (2 * d)) ** 0.5, x_ids="zipf256")
    x, x64 = dev(pr.x, torch.bfloat16)
    Ws, Ws64 = dev(pr.W_self, torch.bfloat16)
    Wn, Wn64 = dev(pr.W_nbr, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    cache = torch.empty(H.hcw_decode_cache_bytes(L, B, n, d), dtype=torch.uint8, device="cuda")
    ys = torch.empty_like(x)
    for t in range(n):
        ys[:, t] = H.hcw_decode_step(x[:, t].contiguous(), Ws, Wn, bias, t, n, cache, flags)
    y, _, _ = H.hcw_stack_fwd(x, Ws, Wn, bias, 0, -1, flags)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    assert rel(host(ys), host(y)) <= TOL_BF16
    ry, _, _ = O.stack_fwd(x64[:2], Ws64, Wn64, pr.bias.astype(np.float64), 0, L, -1, flags,
                           round_bf16=True)
    assert rel(host(ys[:2]), ry) <= TOL_BF16


def test_decode_windows_back_to_back_share_the_cache(H, decode_kernel):
    """A new window restarts at t = 0 on the same rings; its outputs are those
    of a fresh decode on a cache full of garbage, bit for bit (no slot is read
    before it is written)."""
    B, n, d, L, flags = 5, 16, 128, 6, CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=32, w_std=(1 / (2 * d)) ** 0.5)
    Ws = torch.from_numpy(pr.W_self).to(torch.bfloat16).cuda()
    Wn = torch.from_numpy(pr.W_nbr).to(torch.bfloat16).cuda()
    bias = torch.from_numpy(pr.bias).cuda()
    xa = torch.from_numpy(pr.x).to(torch.bfloat16).cuda()
    xb = torch.from_numpy(synth.problem(B, n, d, L=1, seed=33).x).to(torch.bfloat16).cuda()

    def window(x, cache):
        ys = torch.empty_like(x)
        for t in range(n):
            ys[:, t] = H.hcw_decode_step(x[:, t].contiguous(), Ws, Wn, bias, t, n, cache, flags)
        return ys

    nb = H.hcw_decode_cache_bytes(L, B, n, d)
    cache = torch.empty(nb, dtype=torch.uint8, device="cuda")
    window(xa, cache)
    yb = window(xb, cache)
    fresh = window(xb, torch.full((nb,), 0x7F, dtype=torch.uint8, device="cuda"))
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    assert torch.equal(yb, fresh)


def test_stack_fixed_dimension_control(H):
    pr = synth.problem(16, 64, 128, L=6, seed=5, w_std=(1 / 256) ** 0.5)
    got, ref = run_stack(H, pr, torch.bfloat16, 6, 0, dim=0)
    for g, r, what in zip(got, ref, WHAT):
        assert rel(g, r) <= TOL_BF16, what


def test_reach_workload_full_size(H):
    # n = 64, d = 128, six rotated layers, batch 256, non-causal, embedded uniform-16 ids
    w = synth.WORKLOADS["reach_n64_d128"]
    pr = synth.problem(w["B"], w["n"], w["d"], L=w["L"], seed=0, w_std=(1 / 256) ** 0.5,
                       x_ids="uniform16")
    got, ref = run_stack(H, pr, torch.bfloat16, w["L"], 0)
    for g, r, what in zip(got, ref, WHAT):
        assert rel(g, r) <= TOL_BF16, what


@pytest.mark.parametrize("workload", ["charlm_w256_d512", "charlm_w64_d512"])
def test_charlm_full_launch_sampled(H, workload):
    """The char-LM workloads (B = 64, n = 256 or 64, d = 512, 16 causal layers,
    residual, ReLU, bias) in their full launch configuration; the oracle
    recomputes two sampled sequences.  Forward: the device's rows of those
    sequences against the oracle.  Backward: the upstream gradient is zero
    outside them and the device backward sees the oracle's saved activations
    for them (same ReLU decisions), so its weight gradients over the whole
    batch must equal the oracle's over the two sequences, and dx must vanish
    elsewhere."""
    w = synth.WORKLOADS[workload]
    B, n, d, L = w["B"], w["n"], w["d"], w["L"]
    flags = CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=0, w_std=(1 / (2 * d)) ** 0.5, x_ids="zipf256")
    picks = [5, 42]
    mask = np.zeros((B, 1, 1), dtype=np.float32)
    mask[picks] = 1.0
    pr.dy = pr.dy * mask
    x, x64 = dev(pr.x, torch.bfloat16)
    Ws, Ws64 = dev(pr.W_self, torch.bfloat16)
    Wn, Wn64 = dev(pr.W_nbr, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    dy, dy64 = dev(pr.dy, torch.bfloat16)
    y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, 0, -1, flags)
    ry, racts, rzs = O.stack_fwd(x64[picks], Ws64, Wn64, pr.bias.astype(np.float64), 0, L, -1,
                                 flags, round_bf16=True)
    assert rel(host(y)[picks], ry) <= TOL_BF16
    assert rel(host(acts)[:, picks], racts[1:]) <= TOL_BF16
    acts[:, picks] = torch.from_numpy(racts[1:]).to(torch.bfloat16).cuda()
    masks[:, picks] = masks_from_z(rzs).cuda()
    dx, gWs, gWn, gb = H.hcw_stack_bwd(x, acts, masks, dy, Ws, Wn, 0, -1, flags)
    torch.cuda.synchronize()
    rdx, rWs, rWn, rgb = O.stack_bwd(racts, rzs, dy64[picks], Ws64, Wn64, 0, L, -1, flags,
                                     round_bf16=True)
    hdx = host(dx)
    assert rel(hdx[picks], rdx) <= TOL_BF16
    others = np.setdiff1d(np.arange(B), picks)
    assert np.abs(hdx[others]).max() == 0.0
    assert rel(host(gWs), rWs) <= TOL_BF16
    assert rel(host(gWn), rWn) <= TOL_BF16
    assert rel(host(gb), rgb) <= TOL_BF16


def test_scaling_n256_d1024_full_launch_sampled(H):
    """Scaling shape n = 256, d = 1024, 8 rotated non-causal layers, 2^20 tokens
    (4096 sequences) with random weights, in its full launch configuration;
    the oracle recomputes one sequence forward, and the backward (upstream
    gradient zero elsewhere) gives that sequence's weight gradients."""
    w = synth.WORKLOADS["scale_n256_d1024"]
    B, n, d, L = w["B"], w["n"], w["d"], w["L"]
    pick = 1234
    g = torch.Generator().manual_seed(7)
    Ws = (torch.randn((L, d, d), generator=g) * (1 / (2 * d)) ** 0.5).to(torch.bfloat16)
    Wn = (torch.randn((L, d, d), generator=g) * (1 / (2 * d)) ** 0.5).to(torch.bfloat16)
    bias = torch.randn((L, d), generator=g) * 0.1
    x = synth.device_normal((B, n, d), 31, "cuda").to(torch.bfloat16)
    xs = torch.randn((n, d), generator=g).to(torch.bfloat16)     # the sampled sequence
    x[pick] = xs.cuda()
    dys = torch.randn((n, d), generator=g).to(torch.bfloat16)
    dy = torch.zeros((B, n, d), dtype=torch.bfloat16, device="cuda")
    dy[pick] = dys.cuda()
    y, acts, _ = H.hcw_stack_fwd(x, Ws.cuda(), Wn.cuda(), bias.cuda(), 0, -1, 0)
    x64 = xs.double().numpy()[None]
    W64 = (Ws.double().numpy(), Wn.double().numpy())
    ry, racts, rzs = O.stack_fwd(x64, W64[0], W64[1], bias.double().numpy(), 0, L, -1, 0,
                                 round_bf16=True)
    assert rel(host(y[pick])[None], ry) <= TOL_BF16
    assert rel(host(acts[:, pick])[:, None], racts[1:]) <= TOL_BF16
    acts[:, pick] = torch.from_numpy(racts[1:, 0]).to(torch.bfloat16).cuda()
    dx, gWs, gWn, gb = H.hcw_stack_bwd(x, acts, None, dy, Ws.cuda(), Wn.cuda(), 0, -1, 0)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    rdx, rWs, rWn, rgb = O.stack_bwd(racts, rzs, dys.double().numpy()[None], W64[0], W64[1],
                                     0, L, -1, 0, round_bf16=True)
    assert rel(host(dx[pick])[None], rdx) <= TOL_BF16
    others = torch.arange(B, device="cuda") != pick
    assert float(dx[others].float().abs().max()) == 0.0
    assert rel(host(gWs), rWs) <= TOL_BF16
    assert rel(host(gWn), rWn) <= TOL_BF16
    assert rel(host(gb), rgb) <= TOL_BF16


def _block_means(a, l):
    """Mean of a [n, d] sequence over blocks of 2^l consecutive positions,
    broadcast back to every position of the block."""
    n, d = a.shape
    m = a.reshape(n >> l, 1 << l, d).mean(axis=1)
    return np.repeat(m, 1 << l, axis=0)


def _low_means(a, l):
    """Mean over the positions that agree with each position on bits 0..l-1
    (the high bits l..b-1 averaged out), broadcast back."""
    n, d = a.shape
    m = a.reshape(n >> l, 1 << l, d).mean(axis=0)
    return np.tile(m, (n >> l, 1))


@pytest.mark.parametrize("workload", ["scale_n4096_d1024", "scale_n65536_d1024"])
def test_scaling_sweep_identity_weights_any_size(H, workload):
    """Scaling shapes (2^20 tokens, d = 1024, L = log2 n non-causal layers) with
    W_self = W_nbr = I/2: layer l averages each position with its partner
    across bit l, so (the closed form of the pins) layer l's output is the
    mean over the 2^(l+1)-position block, y is the sequence mean, and the
    backward is the same averaging: dx = mean of dy over the sequence, and
    with dz_l the mean of dy over the bits above l, dW_self[l][o][i] =
    sum_t dz_l[t][o] x_l[t][i] and dW_nbr[l][o][i] = sum_t dz_l[t][o]
    x_l[t ^ 2^l][i].  Every product is exact, so the device differs from these
    fp64 values only by its bf16 stores; checked on every position of two
    sequences (upstream gradient on one of them) and sampled weight-gradient
    entries."""
    w = synth.WORKLOADS[workload]
    B, n, d, L = w["B"], w["n"], w["d"], w["L"]
    half = torch.eye(d, dtype=torch.bfloat16, device="cuda") * 0.5
    Ws = half.expand(L, d, d).contiguous()
    x = synth.device_normal((B, n, d), 41, "cuda").to(torch.bfloat16)
    dy = torch.zeros((B, n, d), dtype=torch.bfloat16, device="cuda")
    b0, b1 = 0, B - 1
    dy[b0] = synth.device_normal((n, d), 42, "cuda").to(torch.bfloat16)
    y, acts, _ = H.hcw_stack_fwd(x, Ws, Ws, None, 0, -1, 0)
    dx, dz = H.hcw_stack_bwd_data(None, dy, Ws, Ws, 0, -1, 0)
    gWs, gWn, gb = H.hcw_stack_bwd_weight(x, acts, dz, 0, -1, 0)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    for b in (b0, b1):
        xb = host(x[b])
        assert rel(host(y[b]), _block_means(xb, L)) <= TOL_BF16, b
        for l in (0, L // 2, L - 2):
            assert rel(host(acts[l, b]), _block_means(xb, l + 1)) <= TOL_BF16, (b, l)
    dyb = host(dy[b0])
    assert rel(host(dx[b0]), _block_means(dyb, L)) <= TOL_BF16
    assert float(dx[b1].float().abs().max()) == 0.0
    xb = host(x[b0])
    rng = np.random.default_rng(5)
    for l in (0, 1, L // 2, L - 1):
        xl = _block_means(xb, l)                 # layer l's input
        gl = _low_means(dyb, l + 1)              # gradient at layer l's output (= dz_l)
        part = np.arange(n) ^ (1 << l)
        o = rng.integers(0, d, 16)
        i = rng.integers(0, d, 16)
        ref_s = np.einsum("tk,tk->k", gl[:, o], xl[:, i])
        ref_n = np.einsum("tk,tk->k", gl[:, o], xl[part][:, i])
        got_s = host(gWs[l])[o, i]
        got_n = host(gWn[l])[o, i]
        scale = np.abs(ref_s).max() + np.abs(ref_n).max()
        assert np.abs(got_s - ref_s).max() <= TOL_BF16 * scale, l
        assert np.abs(got_n - ref_n).max() <= TOL_BF16 * scale, l
        assert rel(host(gb[l]), gl.sum(axis=0)) <= TOL_BF16, l


def test_stack_backward_is_the_chain_of_layer_backwards(H):
    """The stack's forward equals hcw_layer_fwd layer by layer and its ReLU masks
    are exactly (z > 0) of those layers; hcw_stack_bwd on its own saved state
    equals hcw_layer_bwd applied layer by layer from the top (dx bit-exact,
    weight and bias gradients up to fp32 summation order): the stack plumbing
    and the fused ReLU gradient add nothing."""
    for flags in (CAUSAL | RESIDUAL | RELU, CAUSAL | RELU, RESIDUAL):
        B, n, d, L = 4, 256, 512, 5
        pr = synth.problem(B, n, d, L=L, seed=4, w_std=(1 / (2 * d)) ** 0.5)
        x, _ = dev(pr.x, torch.bfloat16)
        Ws, _ = dev(pr.W_self, torch.bfloat16)
        Wn, _ = dev(pr.W_nbr, torch.bfloat16)
        dy, _ = dev(pr.dy, torch.bfloat16)
        bias = torch.from_numpy(pr.bias).cuda()
        y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, 3, -1, flags)
        dx, gWs, gWn, gb = H.hcw_stack_bwd(x, acts, masks, dy, Ws, Wn, 3, -1, flags)
        inp, zs = x, []
        for l in range(L):
            out, z = H.hcw_layer_fwd(inp, Ws[l], Wn[l], bias[l], 3 + l, -1, flags, want_z=True)
            assert torch.equal(out, acts[l] if l < L - 1 else y)
            if flags & RELU:
                assert torch.equal(masks_from_z(host(z)).cuda(), masks[l])
            zs.append(z)
            inp = out
        g = dy
        for l in range(L - 1, -1, -1):
            inp = x if l == 0 else acts[l - 1]
            g, a, b, c = H.hcw_layer_bwd(inp, zs[l], g, Ws[l], Wn[l], 3 + l, -1, flags)
            # the stack accumulates each weight gradient over all tokens in one
            # pass, the layer call in token splits: same terms, other fp32 order
            assert rel(host(gWs[l]), host(a)) <= 1e-5 and rel(host(gWn[l]), host(b)) <= 1e-5
            assert rel(host(gb[l]), host(c)) <= 1e-5
        assert torch.equal(g, dx)


def test_split_backward_matches_fused(H):
    flags = CAUSAL | RESIDUAL
    pr = synth.problem(8, 64, 256, L=1, seed=9)
    x, _ = dev(pr.x, torch.bfloat16)
    dy, _ = dev(pr.dy, torch.bfloat16)
    Ws, _ = dev(pr.W_self[0], torch.bfloat16)
    Wn, _ = dev(pr.W_nbr[0], torch.bfloat16)
    dx, gWs, gWn, gb = H.hcw_layer_bwd(x, None, dy, Ws, Wn, 2, -1, flags)
    dx2 = H.hcw_layer_bwd_data(dy, dy, Ws, Wn, 2, -1, flags)
    a, b, c = H.hcw_layer_bwd_weight(x, dy, 2, -1, flags)
    assert torch.equal(dx, dx2) and torch.equal(gWs, a) and torch.equal(gWn, b)
    assert torch.equal(gb, c)


@pytest.mark.parametrize("kernels", ["auto", "resident"])
@pytest.mark.parametrize("dtype,flags", [(torch.bfloat16, CAUSAL | RESIDUAL | RELU),
                                         (torch.bfloat16, CAUSAL), (torch.bfloat16, RELU),
                                         (torch.float32, CAUSAL | RESIDUAL | RELU),
                                         (torch.float32, RESIDUAL)])
def test_stack_backward_halves_match_the_whole(H, dtype, flags, kernels):
    """hcw_stack_bwd_data then hcw_stack_bwd_weight give exactly what
    hcw_stack_bwd gives, and the dz they pass on is each layer's dy * act'(z)
    chain (checked on the top layer, where it is dy masked)."""
    if kernels == "resident" and dtype == torch.float32:
        pytest.skip("the resident kernels are bf16 only")
    d = 64 if dtype == torch.float32 else 256
    B, n, L = 4, 64, 5
    prev = H.hcw_set_stack_kernels(H.HCW_STACK_RESIDENT if kernels == "resident"
                                   else H.HCW_STACK_AUTO)
    try:
        _halves_match_the_whole(H, dtype, flags, d, B, n, L)
    finally:
        H.hcw_set_stack_kernels(prev)


def _halves_match_the_whole(H, dtype, flags, d, B, n, L):
    pr = synth.problem(B, n, d, L=L, seed=21, w_std=(1 / (2 * d)) ** 0.5)
    x, _ = dev(pr.x, dtype)
    Ws, _ = dev(pr.W_self, dtype)
    Wn, _ = dev(pr.W_nbr, dtype)
    dy, _ = dev(pr.dy, dtype)
    bias = torch.from_numpy(pr.bias).cuda()
    y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, 1, -1, flags)
    dx, gWs, gWn, gb = H.hcw_stack_bwd(x, acts, masks, dy, Ws, Wn, 1, -1, flags)
    dx2, dz = H.hcw_stack_bwd_data(masks, dy, Ws, Wn, 1, -1, flags)
    a, b, c = H.hcw_stack_bwd_weight(x, acts, dz, 1, -1, flags)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    assert torch.equal(dx, dx2) and torch.equal(gWs, a) and torch.equal(gWn, b)
    assert torch.equal(gb, c)
    top = dy.clone()
    if flags & RELU:
        bits = masks[L - 1].to(torch.int64) & 0xFFFFFFFF
        keep = ((bits.unsqueeze(-1) >> torch.arange(32, device=bits.device)) & 1).bool()
        top = torch.where(keep.reshape(top.shape), top, torch.zeros_like(top))
    assert torch.equal(dz[L - 1], top)


def test_batched_weight_gradient_against_fp64_sums(H):
    """16 layers whose tiles fill the GPU: one weight-gradient launch for all of
    them (a unit per layer and output tile, self and partner parts together),
    the bias gradient summed inside it.  dW_self[l] = dz_l^T x_l, dW_nbr[l] =
    sum over receiving positions of dz_l,i x_l,i-2^s, dbias[l] = column sums
    of dz_l, recomputed in fp64 from the same bf16 tensors (any summation
    order agrees to fp32 accumulation error)."""
    B, n, d, L = 8, 256, 512, 16
    flags = CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=33, w_std=(1 / (2 * d)) ** 0.5)
    x, _ = dev(pr.x, torch.bfloat16)
    Ws, _ = dev(pr.W_self, torch.bfloat16)
    Wn, _ = dev(pr.W_nbr, torch.bfloat16)
    dy, _ = dev(pr.dy, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, 0, -1, flags)
    dx, dz = H.hcw_stack_bwd_data(masks, dy, Ws, Wn, 0, -1, flags)
    gWs, gWn, gb = H.hcw_stack_bwd_weight(x, acts, dz, 0, -1, flags)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    for l in range(L):
        inp3 = (x if l == 0 else acts[l - 1]).double()
        inp = inp3.reshape(-1, d)
        g = dz[l].reshape(-1, d).double()
        assert rel(host(gb[l]), host(g.sum(0))) <= 1e-5, l
        assert rel(host(gWs[l]), host(g.T @ inp)) <= 1e-5, l
        # causal partner part: positions with bit s set receive from i - 2^s
        s = l % int(np.log2(n))
        recv = torch.tensor([i for i in range(n) if (i >> s) & 1], device="cuda")
        gr = dz[l][:, recv].reshape(-1, d).double()
        xp = inp3[:, recv - (1 << s)].reshape(-1, d)
        assert rel(host(gWn[l]), host(gr.T @ xp)) <= 1e-5, l


def test_batched_weight_gradient_with_shift_layers_against_fp64_sums(H):
    """hcw_stack_bwd_weight_dims on a schedule of shift layers and hypercube
    jumps (the batched launch on SM pairs, shift layers reading their partner
    rows at p - k): every layer's dW_self, dW_nbr and dbias against fp64 sums
    of the same bf16 tensors.  A shift layer by k gives every position p >= k
    of a sequence the partner p - k (Eq. (1)); a jump along dimension s gives
    the positions with bit s set the partner p - 2^s (causal)."""
    B, n, d = 4, 256, 512
    dims = [-1, 7, -1, -3, 5, -1, 4, -64, -1, 2, -255, 1, -1, 0]
    L = len(dims)
    flags = CAUSAL | RESIDUAL | RELU
    pr = synth.problem(B, n, d, L=L, seed=37, w_std=(1 / (2 * d)) ** 0.5)
    x, _ = dev(pr.x, torch.bfloat16)
    Ws, _ = dev(pr.W_self, torch.bfloat16)
    Wn, _ = dev(pr.W_nbr, torch.bfloat16)
    bias = torch.from_numpy(pr.bias).cuda()
    y, acts, masks = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
    g = torch.Generator().manual_seed(41)
    dz = (torch.randn(L, B, n, d, generator=g) * 0.05).to(torch.bfloat16).cuda()
    gWs, gWn, gb = H.hcw_stack_bwd_weight(x, acts, dz, flags=flags, dims=dims)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    for l, s in enumerate(dims):
        inp3 = (x if l == 0 else acts[l - 1]).double()
        g3 = dz[l].double()
        assert rel(host(gb[l]), host(g3.reshape(-1, d).sum(0))) <= 1e-5, l
        assert rel(host(gWs[l]), host(g3.reshape(-1, d).T @ inp3.reshape(-1, d))) <= 1e-5, l
        k = -s if s < 0 else 1 << s
        recv = [i for i in range(n) if (i >= k if s < 0 else (i >> s) & 1)]
        recv = torch.tensor(recv, device="cuda")
        gr = g3[:, recv].reshape(-1, d)
        xp = inp3[:, recv - k].reshape(-1, d)
        assert rel(host(gWn[l]), host(gr.T @ xp)) <= 1e-5, (l, s)


def test_launch_counter_counts_kernels(H):
    pr = synth.problem(2, 16, 64, L=1, seed=1)
    x, _ = dev(pr.x, torch.bfloat16)
    W, _ = dev(pr.W_self[0], torch.bfloat16)
    c0 = H.hcw_launch_count()
    H.hcw_layer_fwd(x, W, W, None, 0)
    assert H.hcw_launch_count() == c0 + 1


# ---------------------------------------------------------------- bounded waits

def test_bounded_wait_reports_timeout_and_context_survives(H):
    assert H.hcw_sync_status() == H.HCW_OK
    H.hcw_selftest_wait(200_000_000)           # nothing arrives: gives up after 0.2 s
    assert H.hcw_sync_status() == H.HCW_ERR_TIMEOUT
    assert H.hcw_sync_status() == H.HCW_OK     # the word was cleared
    pr = synth.problem(4, 16, 64, L=1, seed=1)
    x, x64 = dev(pr.x, torch.bfloat16)
    W, W64 = dev(pr.W_self[0], torch.bfloat16)
    y = H.hcw_layer_fwd(x, W, W, None, 1, -1, CAUSAL)
    torch.cuda.synchronize()
    yr = O.layer_fwd(x64, W64, W64, None, 1, -1, CAUSAL, round_bf16=True)
    assert rel(host(y), yr) <= TOL_BF16
