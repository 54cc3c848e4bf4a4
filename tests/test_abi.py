"""The C-ABI library: it loads without a GPU, exports every entry point that
include/hcw.h declares, and its host-side logic (partner tables, argument
validation) behaves as documented.  No call here launches a kernel."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import oracle as O
from paper_2609_18145_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def hcw():
    _build.build()
    from paper_2609_18145_gb300 import hcw as H
    H.lib()
    return H


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "hcw.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hcw_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_path():
    syms = declared_symbols()
    for name in ("hcw_layer_fwd", "hcw_layer_bwd", "hcw_stack_fwd", "hcw_stack_bwd",
                 "hcw_workspace_bytes", "hcw_partner_table", "hcw_status_string"):
        assert name in syms


def test_library_exports_every_declared_symbol(hcw):
    lib = ctypes.CDLL(hcw.LIB_PATH)
    missing = [s for s in declared_symbols() if not hasattr(lib, s)]
    assert not missing, missing
    assert sorted(hcw.EXPORTED) == declared_symbols()


def test_version_and_status_strings(hcw):
    assert hcw.hcw_version() >= 100
    assert hcw.status_string(0) == "HCW_OK"
    assert hcw.status_string(6) == "HCW_ERR_TIMEOUT"
    assert hcw.status_string(99) == "HCW_ERR_UNKNOWN"


@pytest.mark.parametrize("n", [2, 4, 16, 64, 256, 65536])
@pytest.mark.parametrize("flags", [0, 1])
def test_host_partner_table_matches_oracle(hcw, n, flags):
    b = n.bit_length() - 1
    for layer in list(range(2 * b)) + [1000]:
        got = np.array(hcw.hcw_partner_table(layer, n, flags))
        ref = O.partner_table(layer, -1, n, flags)
        assert np.array_equal(got, ref)
    for dim in range(b):
        got = np.array(hcw.hcw_partner_table(3, n, flags, dim_override=dim))
        assert np.array_equal(got, O.partner_table(3, dim, n, flags))


def test_host_partner_table_rejects(hcw):
    L = hcw.lib()
    buf = (ctypes.c_int * 64)()
    assert L.hcw_partner_table(0, -1, 48, 0, buf) == hcw.HCW_ERR_INVALID_ARG
    assert L.hcw_partner_table(0, 6, 64, 0, buf) == hcw.HCW_ERR_INVALID_ARG
    assert L.hcw_partner_table(-1, -1, 64, 0, buf) == hcw.HCW_ERR_INVALID_ARG
    assert L.hcw_partner_table(0, -1, 64, 0, None) == hcw.HCW_ERR_INVALID_ARG
    assert L.hcw_partner_table(0, -1, 64, 64, buf) == hcw.HCW_ERR_INVALID_ARG


def _fwd(hcw, x, ws, wn, bias, layer, dim, B, n, d, dt, flags, y, z):
    P = ctypes.c_void_p
    return hcw.lib().hcw_layer_fwd(P(x), P(ws), P(wn), P(bias), layer, dim, B, n, d, dt, flags,
                                   P(y), P(z), None)


def test_forward_validation_codes(hcw):
    # fake, never dereferenced addresses: validation returns before any launch
    X, WS, WN, Y = 0x100000, 0x200000, 0x300000, 0x400000
    ok = dict(layer=0, dim=-1, B=4, n=16, d=64, dt=hcw.HCW_BF16, flags=0)

    def call(**kw):
        a = dict(ok, **kw)
        return _fwd(hcw, a.get("x", X), a.get("ws", WS), a.get("wn", WN), a.get("bias"),
                    a["layer"], a["dim"], a["B"], a["n"], a["d"], a["dt"], a["flags"],
                    a.get("y", Y), a.get("z"))

    assert call(n=48) == hcw.HCW_ERR_INVALID_ARG          # n not a power of two
    assert call(n=1) == hcw.HCW_ERR_INVALID_ARG
    assert call(B=-1) == hcw.HCW_ERR_INVALID_ARG
    assert call(layer=-2) == hcw.HCW_ERR_INVALID_ARG
    assert call(dim=4) == hcw.HCW_ERR_INVALID_ARG          # log2 16 = 4 dimensions: 0..3
    assert call(flags=8) == hcw.HCW_ERR_INVALID_ARG
    assert call(dt=7) == hcw.HCW_ERR_INVALID_ARG
    assert call(d=96) == hcw.HCW_ERR_UNSUPPORTED          # bf16 needs d % 64 == 0
    assert call(x=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(y=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(x=X + 8) == hcw.HCW_ERR_ALIGNMENT
    assert call(bias=WS + 4) == hcw.HCW_ERR_ALIGNMENT
    assert call(y=X + 1024) == hcw.HCW_ERR_ALIASING       # y overlaps x
    assert call(z=Y) == hcw.HCW_ERR_ALIASING              # z overlaps y
    assert call(B=0) == hcw.HCW_OK                         # empty batch: nothing to do


def test_backward_validation_codes(hcw):
    P = ctypes.c_void_p
    L = hcw.lib()
    X, DY, WS, WN, DX, GS, GN = (0x100000 * k for k in range(1, 8))
    args = dict(x=X, z=None, dy=DY, ws=WS, wn=WN, layer=0, dim=-1, B=4, n=16, d=32,
                dt=hcw.HCW_F32, flags=0, dx=DX, gs=GS, gn=GN, gb=None, w=None, wsb=0)

    def call(**kw):
        a = dict(args, **kw)
        return L.hcw_layer_bwd(P(a["x"]), P(a["z"]), P(a["dy"]), P(a["ws"]), P(a["wn"]),
                               a["layer"], a["dim"], a["B"], a["n"], a["d"], a["dt"], a["flags"],
                               P(a["dx"]), P(a["gs"]), P(a["gn"]), P(a["gb"]), P(a["w"]),
                               a["wsb"], None)

    need = hcw.hcw_workspace_bytes(4, 16, 32, hcw.HCW_F32, 0)
    assert need > 0
    assert call() == hcw.HCW_ERR_WORKSPACE
    assert call(w=0x900000, wsb=need - 1) == hcw.HCW_ERR_WORKSPACE
    assert call(flags=hcw.HCW_ACT_RELU, w=0x900000, wsb=1 << 30) == hcw.HCW_ERR_INVALID_ARG
    assert call(dx=X, w=0x9000000, wsb=need) == hcw.HCW_ERR_ALIASING
    assert call(gn=GS, w=0x9000000, wsb=need) == hcw.HCW_ERR_ALIASING
    assert call(dx=DX + 4, w=0x9000000, wsb=need) == hcw.HCW_ERR_ALIGNMENT
    assert call(d=0) == hcw.HCW_ERR_INVALID_ARG


def test_weight_gradient_rejects_dbias_over_its_inputs(hcw):
    """The column sums read dz while they write dbias: both weight-gradient
    entry points (with a workspace, and the one without) refuse a dbias that
    overlaps x or dz, before anything launches."""
    P = ctypes.c_void_p
    L = hcw.lib()
    B, n, d = 4, 16, 64
    act = B * n * d * 2
    X, DZ, GS, GN, GB, W = (0x10000000 * k for k in range(1, 7))
    need = hcw.hcw_layer_bwd_weight_workspace_bytes(B, n, d, hcw.HCW_BF16, 0)

    def ws(gb):
        return L.hcw_layer_bwd_weight(P(X), P(DZ), 0, -1, B, n, d, hcw.HCW_BF16, 0, P(GS), P(GN),
                                      P(gb), P(W), need, None)

    def noalloc(gb):
        return L.hcw_layer_bwd_weight_noalloc(P(X), P(DZ), 0, -1, B, n, d, hcw.HCW_BF16, 0,
                                              P(GS), P(GN), P(gb), None)

    for f in (ws, noalloc):
        assert f(X + act - 256) == hcw.HCW_ERR_ALIASING      # inside x
        assert f(DZ) == hcw.HCW_ERR_ALIASING                 # on dz
        assert f(GS + 64) == hcw.HCW_ERR_ALIASING            # inside dW_self
    assert ws(W + 16) == hcw.HCW_ERR_ALIASING                # inside the workspace


def test_workspace_sizes_f32(hcw):
    a = hcw.hcw_workspace_bytes(64, 256, 512, hcw.HCW_F32, 0)
    b = hcw.hcw_workspace_bytes(64, 256, 512, hcw.HCW_F32, hcw.HCW_ACT_RELU)
    assert b - a >= 64 * 256 * 512 * 4            # the masked gradient dz
    s = hcw.hcw_stack_workspace_bytes(64, 256, 512, hcw.HCW_F32, 0, 16)
    assert s >= a + 2 * 64 * 256 * 512 * 4        # gradient buffers between layers
    assert hcw.hcw_workspace_bytes(4, 48, 64, hcw.HCW_F32, 0) == 0   # invalid n


def test_stack_backward_halves_validation_codes(hcw):
    P = ctypes.c_void_p
    L = hcw.lib()
    B, n, d, Ly = 4, 16, 64, 3
    act = B * n * d * 2
    M, DY, WS, WN, DX, DZ, W = (0x10000000 * k for k in range(1, 8))
    flags = hcw.HCW_CAUSAL | hcw.HCW_RESIDUAL | hcw.HCW_ACT_RELU
    need = hcw.hcw_stack_bwd_data_workspace_bytes(B, n, d, hcw.HCW_BF16, flags, Ly)
    assert need > 0
    args = dict(m=M, dy=DY, ws=WS, wn=WN, dx=DX, dz=DZ, w=W, wsb=need, flags=flags, Ly=Ly)

    def data(**kw):
        a = dict(args, **kw)
        return L.hcw_stack_bwd_data(P(a["m"]), P(a["dy"]), P(a["ws"]), P(a["wn"]), 0, a["Ly"],
                                    -1, B, n, d, hcw.HCW_BF16, a["flags"], P(a["dx"]),
                                    P(a["dz"]), P(a["w"]), a["wsb"], None)

    assert data(m=0) == hcw.HCW_ERR_INVALID_ARG            # ReLU needs the masks
    assert data(dz=0) == hcw.HCW_ERR_INVALID_ARG
    assert data(Ly=0) == hcw.HCW_ERR_INVALID_ARG
    assert data(wsb=need - 1) == hcw.HCW_ERR_WORKSPACE
    assert data(dz=DZ + 8) == hcw.HCW_ERR_ALIGNMENT
    assert data(dx=DZ + (Ly - 1) * act) == hcw.HCW_ERR_ALIASING   # dx inside dz
    assert data(w=DZ) == hcw.HCW_ERR_ALIASING               # workspace over dz
    assert data(dz=DY) == hcw.HCW_ERR_ALIASING              # dz over dy

    wneed = hcw.hcw_stack_bwd_weight_workspace_bytes(B, n, d, hcw.HCW_BF16, flags, Ly)
    assert wneed > 0
    X, A, GS, GN, GB = (0x20000000 * k for k in range(1, 6))

    def weight(**kw):
        a = dict(dict(x=X, acts=A, dz=DZ, gs=GS, gn=GN, gb=GB, w=W, wsb=wneed), **kw)
        return L.hcw_stack_bwd_weight(P(a["x"]), P(a["acts"]), P(a["dz"]), 0, Ly, -1, B, n, d,
                                      hcw.HCW_BF16, flags, P(a["gs"]), P(a["gn"]), P(a["gb"]),
                                      P(a["w"]), a["wsb"], None)

    assert weight(acts=0) == hcw.HCW_ERR_INVALID_ARG        # L > 1 needs the layer inputs
    assert weight(wsb=wneed - 1) == hcw.HCW_ERR_WORKSPACE
    assert weight(gn=GS) == hcw.HCW_ERR_ALIASING
    assert weight(gs=DZ) == hcw.HCW_ERR_ALIASING            # gradient written over dz
    assert weight(gb=GB + 4) == hcw.HCW_ERR_ALIGNMENT


def test_stack_workspace_is_the_sum_of_its_parts(hcw):
    for dt, flags in ((hcw.HCW_BF16, 7), (hcw.HCW_BF16, 1), (hcw.HCW_F32, 7)):
        B, n, d, Ly = 64, 256, 512, 16
        total = hcw.hcw_stack_workspace_bytes(B, n, d, dt, flags, Ly)
        es = 2 if dt == hcw.HCW_BF16 else 4
        parts = (Ly * B * n * d * es + hcw.hcw_stack_bwd_data_workspace_bytes(B, n, d, dt, flags, Ly)
                 + hcw.hcw_stack_bwd_weight_workspace_bytes(B, n, d, dt, flags, Ly))
        assert parts <= total <= parts + 512


@pytest.mark.timeout(60)
def test_workspace_query_terminates_for_wide_layers(hcw):
    # more output tiles than SMs: the split search must stop at one split per part
    for d in (2048, 4096, 8192):
        a = hcw.hcw_layer_bwd_weight_workspace_bytes(1 << 20, 4, d, hcw.HCW_BF16, 0)
        b = hcw.hcw_workspace_bytes(1 << 20, 4, d, hcw.HCW_BF16, hcw.HCW_CAUSAL)
        assert a > 0 and b > 0


def test_stack_kernel_selection_is_a_process_setting(hcw):
    lib = hcw.lib()
    prev = lib.hcw_set_stack_kernels(hcw.HCW_STACK_RESIDENT)
    try:
        assert prev in (hcw.HCW_STACK_AUTO, hcw.HCW_STACK_RESIDENT, hcw.HCW_STACK_STREAMING)
        assert lib.hcw_set_stack_kernels(hcw.HCW_STACK_STREAMING) == hcw.HCW_STACK_RESIDENT
        assert lib.hcw_set_stack_kernels(7) == -1          # unknown: unchanged
        assert lib.hcw_set_stack_kernels(-1) == -1
        # streaming only: every bf16 shape; resident where the shape fits
        assert lib.hcw_stack_kernels_used(64, 256, 512, hcw.HCW_BF16) == hcw.HCW_STACK_STREAMING
        lib.hcw_set_stack_kernels(hcw.HCW_STACK_RESIDENT)
        assert lib.hcw_stack_kernels_used(64, 256, 512, hcw.HCW_BF16) == hcw.HCW_STACK_RESIDENT
        assert lib.hcw_stack_kernels_used(1, 256, 128, hcw.HCW_BF16) == hcw.HCW_STACK_RESIDENT
        assert lib.hcw_stack_kernels_used(64, 512, 512, hcw.HCW_BF16) == hcw.HCW_STACK_STREAMING
        assert lib.hcw_stack_kernels_used(64, 256, 1024, hcw.HCW_BF16) == hcw.HCW_STACK_STREAMING
        assert lib.hcw_stack_kernels_used(64, 256, 384, hcw.HCW_BF16) == hcw.HCW_STACK_STREAMING
        assert lib.hcw_stack_kernels_used(3, 64, 512, hcw.HCW_BF16) == hcw.HCW_STACK_STREAMING
        assert lib.hcw_stack_kernels_used(64, 256, 512, hcw.HCW_F32) == hcw.HCW_STACK_STREAMING
        assert lib.hcw_stack_kernels_used(64, 48, 512, hcw.HCW_BF16) == -1
        lib.hcw_set_stack_kernels(hcw.HCW_STACK_STREAMING)
        assert lib.hcw_set_stack_kernels(hcw.HCW_STACK_AUTO) == hcw.HCW_STACK_STREAMING
        with pytest.raises(ValueError):
            hcw.hcw_set_stack_kernels(3)
    finally:
        lib.hcw_set_stack_kernels(prev)


def test_schedule_entry_points_reject_bad_dims_before_any_launch(hcw):
    """hcw_stack_fwd_dims / hcw_stack_bwd_dims check the schedule (per layer a
    cube dimension in [0, log2 n), or a shift -k with 1 <= k < n) before
    touching a buffer."""
    lib = hcw.lib()
    fake = ctypes.c_void_p(256)   # never dereferenced: the schedule check comes first
    B, n, d, L = 2, 64, 128, 4
    before = hcw.hcw_launch_count()
    # a valid schedule with near (-1) and a shift of 63 gets past the check and
    # stops at the missing workspace
    ok = (ctypes.c_int * L)(0, -1, 5, -63)
    rc = lib.hcw_stack_fwd_dims(fake, fake, fake, None, ctypes.cast(ok, ctypes.c_void_p), L, B, n,
                                d, hcw.HCW_BF16, 0, fake, fake, None, None, 0, None)
    assert rc == hcw.HCW_ERR_WORKSPACE
    for dims in (None, [0, 1, 6, 2], [0, -64, 2, 3], [5, 4, 3, 64]):
        arr = None if dims is None else (ctypes.c_int * L)(*dims)
        ptr = None if arr is None else ctypes.cast(arr, ctypes.c_void_p)
        rc = lib.hcw_stack_fwd_dims(fake, fake, fake, None, ptr, L, B, n, d, hcw.HCW_BF16, 0,
                                    fake, fake, None, None, 0, None)
        assert rc == hcw.HCW_ERR_INVALID_ARG, dims
        rc = lib.hcw_stack_bwd_dims(fake, fake, None, fake, fake, fake, ptr, L, B, n, d,
                                    hcw.HCW_BF16, 0, fake, fake, fake, None, None, 0, None)
        assert rc == hcw.HCW_ERR_INVALID_ARG, dims
        rc = lib.hcw_stack_bwd_weight_dims(fake, fake, fake, ptr, L, B, n, d, hcw.HCW_BF16, 0,
                                           fake, fake, None, None, 0, None)
        assert rc == hcw.HCW_ERR_INVALID_ARG, dims
        rc = lib.hcw_stack_train_step_dims(fake, fake, fake, None, fake, ptr, L, B, n, d,
                                           hcw.HCW_BF16, 0, fake, fake, fake, fake, fake, fake,
                                           None, None, 0, None)
        assert rc == hcw.HCW_ERR_INVALID_ARG, dims
    assert hcw.hcw_launch_count() == before
    with pytest.raises(ValueError):
        hcw._dims_array([0, 1, 2], 4)


def test_small_d_weight_gradient_workspace_holds_the_split_partials(hcw):
    """Few output tiles (d = 128 or 256): the layers' weight gradients split the
    token range over one launch, so the workspace holds fp32 partial weight
    tiles and dbias partials of every layer of the launch; it grows with the
    layer count (up to 16 a launch), and the training step's workspace holds
    it."""
    B, n = 256, 64
    for d in (128, 256):
        one = hcw.hcw_stack_bwd_weight_workspace_bytes(B, n, d, hcw.HCW_BF16, 7, 1)
        six = hcw.hcw_stack_bwd_weight_workspace_bytes(B, n, d, hcw.HCW_BF16, 7, 6)
        sixteen = hcw.hcw_stack_bwd_weight_workspace_bytes(B, n, d, hcw.HCW_BF16, 7, 16)
        assert 0 < one <= six <= sixteen
        # at least two splits of two d x d fp32 parts per layer
        assert six >= 6 * 2 * 2 * d * d * 4
        step = hcw.hcw_stack_train_step_workspace_bytes(B, n, d, hcw.HCW_BF16, 7, 6)
        assert step >= six


def test_decode_cache_is_bounded_by_the_link_distances(hcw):
    """Sec. 6: a layer keeps only the last k inputs it links to.  The rings
    hold sum_l (k_l + 1) slots of B x d bf16 (the input at t goes to a slot
    apart from the one of t - k), not the window: the rotated stack at n = 256
    keeps 2 x (1 + 2 + ... + 128) + 16 = 526 slots instead of 16 x 256."""
    B, d = 3, 64
    assert hcw.hcw_decode_cache_bytes(16, B, 256, d) == 526 * B * d * 2
    hy = [-1, 7, -1, -1, 5, -1, 4, -1, -1, 2, -1, 1, -1, 0]   # 8 near + jumps 128 .. 1
    assert hcw.hcw_decode_cache_bytes(len(hy), B, 256, d, dims=hy) == (8 + 183 + 14) * B * d * 2
    assert hcw.hcw_decode_cache_bytes(3, B, 256, d, dims=[0, -255, 2]) == (2 + 256 + 5) * B * d * 2
    assert hcw.hcw_decode_cache_bytes(2, B, 48, d) == 0              # n not a power of two


def test_decode_step_rejects_bad_arguments_before_any_launch(hcw):
    lib = hcw.lib()
    fake = ctypes.c_void_p(256)
    B, n, d, L = 2, 64, 128, 4
    before = hcw.hcw_launch_count()

    def step(t, flags, d=d, y=ctypes.c_void_p(1 << 20)):
        return lib.hcw_decode_step(fake, fake, fake, None, None, 0, L, t, B, n, d, flags, fake, y,
                                   None)

    assert step(0, 0) == hcw.HCW_ERR_INVALID_ARG             # decoding needs the causal rule
    assert step(n, hcw.HCW_CAUSAL) == hcw.HCW_ERR_INVALID_ARG
    assert step(-1, hcw.HCW_CAUSAL) == hcw.HCW_ERR_INVALID_ARG
    assert step(0, hcw.HCW_CAUSAL, d=2048) == hcw.HCW_ERR_UNSUPPORTED   # one cluster: d <= 1024
    assert step(0, hcw.HCW_CAUSAL, y=ctypes.c_void_p(264)) == hcw.HCW_ERR_ALIGNMENT
    assert step(0, hcw.HCW_CAUSAL, y=fake) == hcw.HCW_ERR_ALIASING       # y_t on the cache
    assert hcw.hcw_launch_count() == before


def test_block_workspace_size_and_validation(hcw):
    """The block step validates sizes, pointers, alignment and the workspace
    before any launch."""
    assert hcw.hcw_block_workspace_bytes(2, 16, 64, 128, 11, 2) > 0
    assert hcw.hcw_block_workspace_bytes(2, 12, 64, 128, 11, 2) == 0    # n not a power of two
    assert hcw.hcw_block_workspace_bytes(2, 16, 96, 128, 11, 2) == 0    # d not a multiple of 64
    assert hcw.hcw_block_workspace_bytes(2, 16, 64, 12, 11, 2) == 0     # h not a multiple of 8
    assert hcw.hcw_block_workspace_bytes(2, 16, 64, 128, 1, 2) == 0     # V < 2
    lib = hcw.lib()
    fake = 1 << 20
    P = hcw._BlockPtrs(*([fake] * len(hcw.BLOCK_FIELDS)))
    G = hcw._BlockPtrs(*([fake + (1 << 16)] * len(hcw.BLOCK_FIELDS)))
    ws_b = hcw.hcw_block_workspace_bytes(2, 16, 64, 128, 11, 2)
    before = hcw.hcw_launch_count()

    def step(P=P, G=G, d=64, ids=ctypes.c_void_p(fake), loss=ctypes.c_void_p(fake), ws=ws_b):
        return lib.hcw_block_step(ids, ctypes.byref(P), ctypes.byref(G), 2, 16, d, 128, 11, 2,
                                  loss, ctypes.c_void_p(1 << 30), ws, None)

    assert lib.hcw_block_step(ctypes.c_void_p(fake), None, ctypes.byref(G), 2, 16, 64, 128, 11, 2,
                              ctypes.c_void_p(fake), ctypes.c_void_p(1 << 30), ws_b,
                              None) == hcw.HCW_ERR_INVALID_ARG
    assert step(d=2048) == hcw.HCW_ERR_UNSUPPORTED           # LayerNorm rows: d <= 1024
    assert step(ids=None) == hcw.HCW_ERR_INVALID_ARG
    Pbad = hcw._BlockPtrs(*([fake] * 15 + [fake + 4]))
    assert step(P=Pbad) == hcw.HCW_ERR_ALIGNMENT
    assert step(ws=ws_b - 256) == hcw.HCW_ERR_WORKSPACE
    assert hcw.hcw_launch_count() == before


def test_gemm_validation_codes(hcw):
    """hcw_gemm_bf16 rejects bad sizes, flags, a misaligned workspace and a C
    that overlaps an operand or the workspace before anything launches."""
    P = ctypes.c_void_p
    L = hcw.lib()
    M, N, K = 256, 512, 128
    A, B, C, W = (0x1000000 * k for k in range(1, 5))

    def call(M=M, N=N, K=K, a=A, ta=0, b=B, tb=1, c=C, w=None, wsb=0):
        return L.hcw_gemm_bf16(M, N, K, P(a), ta, P(b), tb, P(c), P(w) if w else None, wsb,
                               None)

    assert call(M=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(K=-1) == hcw.HCW_ERR_INVALID_ARG
    assert call(a=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(c=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(ta=2) == hcw.HCW_ERR_INVALID_ARG
    assert call(w=W + 8, wsb=1 << 20) == hcw.HCW_ERR_ALIGNMENT
    assert call(c=A + M * K * 2 - 4) == hcw.HCW_ERR_ALIASING      # C's start inside A
    assert call(c=B - 64) == hcw.HCW_ERR_ALIASING                 # C's end inside B
    assert call(w=C + 256, wsb=1 << 20) == hcw.HCW_ERR_ALIASING   # workspace inside C


def test_batched_gemm_validation_codes(hcw):
    """hcw_gemm_bf16_batched rejects bad sizes, strides and a C that overlaps
    an operand's span before anything launches."""
    P = ctypes.c_void_p
    L = hcw.lib()
    M, N, K, nb = 256, 512, 128, 3
    A, B, C = (0x10000000 * k for k in range(1, 4))

    def call(M=M, N=N, K=K, a=A, sa=M * K, b=B, sb=N * K, c=C, batch=nb):
        return L.hcw_gemm_bf16_batched(M, N, K, P(a), sa, P(b), sb, P(c), batch, None)

    before = hcw.hcw_launch_count()
    assert call(batch=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(N=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(sa=-1) == hcw.HCW_ERR_INVALID_ARG
    assert call(b=0) == hcw.HCW_ERR_INVALID_ARG
    assert call(c=A + (nb - 1) * M * K * 2) == hcw.HCW_ERR_ALIASING   # C inside A's last product
    assert call(c=B - 64) == hcw.HCW_ERR_ALIASING                      # C's end inside B
    assert hcw.hcw_launch_count() == before


def test_gemm_workspace_sizes(hcw):
    """A weight-gradient shape (few output tiles, long K) asks for a K split;
    a short K or a wide output asks for none."""
    s = hcw.hcw_gemm_workspace_bytes(512, 1024, 16384)
    assert s > 0 and s % (512 * 1024 * 4) == 0
    assert hcw.hcw_gemm_workspace_bytes(16384, 1024, 512) == 0
    assert hcw.hcw_gemm_workspace_bytes(256, 256, 128) == 0
    assert hcw.hcw_gemm_workspace_bytes(0, 256, 128) == 0


def test_decode_kernel_switch(hcw):
    """hcw_set_decode_kernel returns the previous contraction and refuses an
    unknown one without changing it."""
    L = hcw.lib()
    prev = L.hcw_set_decode_kernel(hcw.HCW_DECODE_TCGEN05)
    try:
        assert prev in (hcw.HCW_DECODE_WARP_MMA, hcw.HCW_DECODE_TCGEN05)
        assert L.hcw_set_decode_kernel(7) == -1
        assert L.hcw_set_decode_kernel(hcw.HCW_DECODE_WARP_MMA) == hcw.HCW_DECODE_TCGEN05
    finally:
        L.hcw_set_decode_kernel(prev)


def test_compute_calls_take_device_tensors_only(hcw):
    """No CPU fallback: the compute entry points of the binding reject host
    tensors before anything reaches the library."""
    import torch
    x = torch.zeros(2, 16, 64, dtype=torch.bfloat16)
    W = torch.zeros(1, 64, 64, dtype=torch.bfloat16)
    before = hcw.hcw_launch_count()
    calls = (lambda: hcw.hcw_layer_fwd(x, W[0], W[0]),
             lambda: hcw.hcw_stack_fwd(x, W, W),
             lambda: hcw.hcw_stack_train_step(x, W, W, None, x),
             lambda: hcw.hcw_stack_bwd_weight(x, None, W.reshape(1, 1, 64, 64)))
    for call in calls:
        with pytest.raises(ValueError, match="CUDA tensors"):
            call()
    assert hcw.hcw_launch_count() == before
