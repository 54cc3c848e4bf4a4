"""hcw_stack_train_step (the forward and the backward of a stack in one call)
against the separate hcw_stack_fwd and hcw_stack_bwd calls, bit for bit, and
against the fp64 oracle.  Where the shape allows it (bf16, rotated schedule,
pairs of SMs, up to 16 layers) the step runs the forward and the input
gradient as one launch; the others run the two calls, which is checked too."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_18145_gb300 import synth

pytestmark = pytest.mark.gpu

CAUSAL, RESIDUAL, RELU = 1, 2, 4
TOL_BF16 = 2e-2


@pytest.fixture(scope="module")
def H():
    from paper_2609_18145_gb300 import hcw
    hcw.lib()
    return hcw


def problem(B, n, d, L, seed):
    pr = synth.problem(B, n, d, L=L, seed=seed, w_std=(1 / (2 * d)) ** 0.5)
    t = lambda a: synth.to_bf16_exact(a)[0].cuda()
    return pr, t(pr.x), t(pr.W_self), t(pr.W_nbr), t(pr.dy), torch.from_numpy(pr.bias).cuda()


def separate(H, x, Ws, Wn, bias, dy, layer0, flags):
    y, acts, masks = H.hcw_stack_fwd(x, Ws, Wn, bias, layer0, -1, flags)
    dx, gWs, gWn, gb = H.hcw_stack_bwd(x, acts, masks, dy, Ws, Wn, layer0, -1, flags)
    return y, acts, masks, dx, gWs, gWn, gb


CASES = [
    # B, n, d, L, layer0, flags
    (64, 256, 512, 16, 0, CAUSAL | RESIDUAL | RELU),   # the timed workload
    (4, 256, 512, 5, 3, CAUSAL | RESIDUAL | RELU),
    (4, 256, 512, 3, 0, CAUSAL | RELU),
    (4, 256, 512, 4, 1, RESIDUAL),
    (2, 128, 256, 1, 0, CAUSAL | RESIDUAL | RELU),     # one layer
    (6, 64, 512, 7, 2, RESIDUAL | RELU),               # non-causal
    (3, 64, 512, 2, 0, CAUSAL | RESIDUAL | RELU),
    (8, 64, 128, 6, 0, RESIDUAL | RELU),               # d = 128: 128-column tiles on pairs
    (32, 64, 128, 6, 1, CAUSAL | RESIDUAL | RELU),
    (2, 64, 128, 3, 0, RESIDUAL | RELU),               # 128 tokens: the two calls
    (4, 64, 192, 3, 0, CAUSAL | RESIDUAL | RELU),      # 64-column tiles: the two calls
    # enough layers for the batched weight gradient on SM pairs, which then
    # starts behind the fused launch and waits on its completion counters
    (4, 256, 512, 12, 5, CAUSAL | RESIDUAL | RELU),
    (2, 512, 512, 12, 0, RESIDUAL | RELU),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B%d_n%d_d%d_L%d_l%d_f%d" % c)
def test_train_step_equals_forward_then_backward(H, case):
    B, n, d, L, layer0, flags = case
    _, x, Ws, Wn, dy, bias = problem(B, n, d, L, seed=11)
    got = H.hcw_stack_train_step(x, Ws, Wn, bias, dy, layer0, -1, flags)
    ref = separate(H, x, Ws, Wn, bias, dy, layer0, flags)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    for name, a, b in zip(("y", "acts", "masks", "dx", "dW_self", "dW_nbr", "dbias"), got, ref):
        if a is None or b is None:
            assert a is None and b is None, name
            continue
        assert torch.equal(a, b), name


def test_train_step_forward_matches_the_oracle(H):
    """The step's forward (y and every saved layer input) against the oracle's
    stack forward in bf16-storage mode; its backward equals the separate
    backward call bit for bit (above), which the stack parity tests hold to
    the oracle."""
    B, n, d, L = 2, 256, 512, 4
    flags = CAUSAL | RESIDUAL | RELU
    pr, x, Ws, Wn, dy, bias = problem(B, n, d, L, seed=12)
    y, acts, masks, dx, gWs, gWn, gb = H.hcw_stack_train_step(x, Ws, Wn, bias, dy, 0, -1, flags)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    ex = lambda t: t.double().cpu().numpy()
    ry, racts, rzs = O.stack_fwd(ex(x), ex(Ws), ex(Wn), pr.bias.astype(np.float64), 0, L, -1,
                                 flags, round_bf16=True)
    rel = lambda a, b: float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))
    assert rel(ex(y.float()), ry) <= TOL_BF16
    for l in range(L - 1):
        assert rel(ex(acts[l].float()), racts[l + 1]) <= TOL_BF16, l


def test_train_step_rejects_overlapping_dy(H):
    B, n, d, L = 4, 256, 512, 2
    flags = CAUSAL | RESIDUAL | RELU
    _, x, Ws, Wn, dy, bias = problem(B, n, d, L, seed=13)
    y = torch.empty_like(x)
    with pytest.raises(H.HcwError) as e:
        H.hcw_stack_train_step(x, Ws, Wn, bias, y, 0, -1, flags, y=y)
    assert e.value.status == H.HCW_ERR_ALIASING


DIMS_CASES = [
    # B, n, d, flags, dims (-k: a shift of Eq. (1) by k)
    (4, 256, 512, CAUSAL | RESIDUAL | RELU, [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0]),
    (2, 256, 512, RESIDUAL, [-3, -64, 2, -127, -1, 5, -200, 0, -1, 7, -2, 3, -130, -255]),
    (4, 128, 512, CAUSAL | RESIDUAL | RELU, [-1, 6, -2, 3, -127, 0, 5, -64, 1, -1, 4, 2]),
    (3, 128, 512, CAUSAL | RESIDUAL | RELU, [-1, 6, -2, 3]),   # 384 tokens: the two calls
    (8, 64, 128, CAUSAL | RESIDUAL | RELU, [-1, 5, -1, 4]),    # n = 64: the two calls
]


@pytest.mark.parametrize("case", DIMS_CASES, ids=lambda c: "B%d_n%d_d%d_f%d_L%d" % (
    c[0], c[1], c[2], c[3], len(c[4])))
def test_train_step_with_a_schedule_equals_the_two_calls(H, case):
    """hcw_stack_train_step_dims (shift layers in the one-launch forward +
    input gradient where the shape allows it) against hcw_stack_fwd_dims then
    hcw_stack_bwd_dims, bit for bit, and its forward against the oracle."""
    B, n, d, flags, dims = case
    L = len(dims)
    pr, x, Ws, Wn, dy, bias = problem(B, n, d, L, seed=13)
    got = H.hcw_stack_train_step(x, Ws, Wn, bias, dy, flags=flags, dims=dims)
    y, acts, masks = H.hcw_stack_fwd_dims(x, Ws, Wn, bias, dims, flags)
    ref = (y, acts, masks) + tuple(H.hcw_stack_bwd_dims(x, acts, masks, dy, Ws, Wn, dims, flags))
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    for name, a, b in zip(("y", "acts", "masks", "dx", "dW_self", "dW_nbr", "dbias"), got, ref):
        if a is None or b is None:
            assert a is None and b is None, name
            continue
        assert torch.equal(a, b), name
    x64 = x.double().cpu().numpy()
    ry, _, _ = O.stack_fwd(x64, Ws.double().cpu().numpy(), Wn.double().cpu().numpy(),
                           pr.bias.astype(np.float64), 0, L, -1, flags, round_bf16=True,
                           dims=dims)
    err = np.abs(got[0].double().cpu().numpy() - ry).max() / max(np.abs(ry).max(), 1e-30)
    assert err <= TOL_BF16, err
