"""hcw_layer_bwd_weight_noalloc on the GPU: the weight gradient for callers
that cannot allocate device memory (a host that lends only its own input and
output buffers, or code that must not call an allocator).  It keeps its
scratch in a fixed array inside the library instead of a caller-provided
workspace, so it is checked here against hcw_layer_bwd_weight, which takes a
workspace, on several calls in a row: later calls find earlier calls'
leftovers in the shared array.  This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_18145_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = 1e-4          # relative tolerance of the bf16 weight-gradient parity tests
TOL_F32 = 1e-5      # and of the fp32 path
CAUSAL, RESIDUAL = 1, 2


def _rel(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    assert np.isfinite(a).all()
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


def _case(B, n, d, seed, dtype):
    pr = synth.problem(B, n, d, L=1, seed=seed, w_std=(1 / (2 * d)) ** 0.5)
    x = torch.from_numpy(pr.x).to(dtype).cuda()
    dz = torch.from_numpy(pr.dy).to(dtype).cuda()
    return x, dz


def _noalloc(H, x, dz, layer, flags):
    B, n, d = x.shape
    dt = H.HCW_BF16 if x.dtype == torch.bfloat16 else H.HCW_F32
    gs = torch.full((d, d), float("nan"), device="cuda")
    gn = torch.full((d, d), float("nan"), device="cuda")
    gb = torch.full((d,), float("nan"), device="cuda")
    P = ctypes.c_void_p
    rc = H.lib().hcw_layer_bwd_weight_noalloc(
        P(x.data_ptr()), P(dz.data_ptr()), layer, -1, B, n, d, dt, flags, P(gs.data_ptr()),
        P(gn.data_ptr()), P(gb.data_ptr()), P(torch.cuda.current_stream().cuda_stream))
    assert rc == H.HCW_OK, H.status_string(rc)
    return gs, gn, gb


def test_noalloc_weight_gradient_matches_workspace_version_twice():
    from paper_2609_18145_gb300 import hcw as H
    H.lib()
    calls = [
        # the timed workload's shape first (split-K slabs and column sums
        # fill the shared array), then a smaller, different one, then the
        # large shape again with another seed and layer: it reads slabs the
        # earlier calls left dirty; last, one fp32 case, whose column sums use
        # the same array
        ((64, 256, 512, 1, torch.bfloat16), 3, CAUSAL | RESIDUAL, TOL),
        ((8, 64, 128, 2, torch.bfloat16), 1, 0, TOL),
        ((64, 256, 512, 5, torch.bfloat16), 6, CAUSAL, TOL),
        ((16, 64, 96, 4, torch.float32), 2, 0, TOL_F32),
    ]
    for (B, n, d, seed, dtype), layer, flags, tol in calls:
        x, dz = _case(B, n, d, seed, dtype)
        got = _noalloc(H, x, dz, layer, flags)
        ref = H.hcw_layer_bwd_weight(x, dz, layer, -1, flags)
        torch.cuda.synchronize()
        assert H.hcw_sync_status() == H.HCW_OK
        for g, r in zip(got, ref):
            assert _rel(g, r) <= tol


def test_noalloc_rejects_sizes_beyond_its_scratch():
    """Sizes beyond the fixed scratch are rejected before any pointer is
    looked at: every pointer here is NULL, so nothing can launch whatever the
    outcome."""
    from paper_2609_18145_gb300 import hcw as H
    big = (1 << 20, 4, 4096)     # needs far more than the 32 MiB of fixed scratch
    assert H.hcw_layer_bwd_weight_workspace_bytes(*big, H.HCW_BF16, 0) > (32 << 20)
    rc = H.lib().hcw_layer_bwd_weight_noalloc(None, None, 0, -1, *big, H.HCW_BF16, 0, None,
                                              None, None, None)
    assert rc == H.HCW_ERR_WORKSPACE
