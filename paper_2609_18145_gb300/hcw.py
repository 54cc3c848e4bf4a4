"""Thin ctypes binding of libhcw (include/hcw.h), same names as the C ABI.

Argument marshalling only: every step of the mixing path runs in the CUDA
kernels of libhcw.  torch supplies device memory and the current stream.
There is no fallback: if libhcw.so is missing or a call fails, an exception
is raised.

Layouts (Sec. 3.1 wiring, Eq. (1) maps): activations [B, n, d] contiguous;
weights [d_out, d_in] acting on column vectors (stacks: [L, d, d]); bias and
weight gradients fp32.  dtype follows x: torch.bfloat16 -> HCW_BF16,
torch.float32 -> HCW_F32.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

HCW_OK = 0
HCW_ERR_INVALID_ARG = 1
HCW_ERR_UNSUPPORTED = 2
HCW_ERR_ALIGNMENT = 3
HCW_ERR_ALIASING = 4
HCW_ERR_CUDA = 5
HCW_ERR_TIMEOUT = 6
HCW_ERR_WORKSPACE = 7

HCW_STACK_AUTO = 0
HCW_STACK_RESIDENT = 1
HCW_STACK_STREAMING = 2
HCW_DECODE_WARP_MMA = 0
HCW_DECODE_TCGEN05 = 1

HCW_BF16 = 0
HCW_F32 = 1

HCW_CAUSAL = 1
HCW_RESIDUAL = 2
HCW_ACT_RELU = 4

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libhcw.so")

_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_U = ctypes.c_uint
_SZ = ctypes.c_size_t
_LL = ctypes.c_longlong

_SIGNATURES = {
    "hcw_version": ([], _I),
    "hcw_status_string": ([_I], ctypes.c_char_p),
    "hcw_partner_table": ([_I, _I, _I, _U, _P], _I),
    "hcw_partner_table_device": ([_I, _I, _I, _U, _P, _P], _I),
    "hcw_layer_fwd": ([_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P], _I),
    "hcw_workspace_bytes": ([_I, _I, _I, _I, _U], _SZ),
    "hcw_layer_bwd": ([_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _P,
                       _SZ, _P], _I),
    "hcw_layer_bwd_data": ([_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P], _I),
    "hcw_layer_bwd_weight_workspace_bytes": ([_I, _I, _I, _I, _U], _SZ),
    "hcw_layer_bwd_weight": ([_P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _SZ, _P], _I),
    "hcw_layer_bwd_weight_noalloc": ([_P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P], _I),
    "hcw_launch_count": ([], ctypes.c_ulonglong),
    "hcw_stack_fwd": ([_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _SZ,
                       _P], _I),
    "hcw_stack_fwd_dims": ([_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _SZ,
                            _P], _I),
    "hcw_stack_bwd_dims": ([_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P,
                            _P, _SZ, _P], _I),
    "hcw_stack_fwd_workspace_bytes": ([_I, _I, _I, _I, _U, _I], _SZ),
    "hcw_stack_workspace_bytes": ([_I, _I, _I, _I, _U, _I], _SZ),
    "hcw_stack_bwd_data": ([_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _SZ,
                            _P], _I),
    "hcw_stack_bwd_data_workspace_bytes": ([_I, _I, _I, _I, _U, _I], _SZ),
    "hcw_stack_bwd_weight": ([_P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _SZ,
                              _P], _I),
    "hcw_stack_bwd_weight_workspace_bytes": ([_I, _I, _I, _I, _U, _I], _SZ),
    "hcw_stack_bwd": ([_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P,
                       _P, _P, _SZ, _P], _I),
    "hcw_stack_train_step": ([_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P,
                              _P, _P, _P, _P, _P, _SZ, _P], _I),
    "hcw_stack_train_step_workspace_bytes": ([_I, _I, _I, _I, _U, _I], _SZ),
    "hcw_stack_bwd_weight_dims": ([_P, _P, _P, _P, _I, _I, _I, _I, _I, _U, _P, _P, _P, _P, _SZ,
                                   _P], _I),
    "hcw_stack_train_step_dims": ([_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _U, _P, _P, _P,
                                   _P, _P, _P, _P, _P, _SZ, _P], _I),
    "hcw_decode_step": ([_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _U, _P, _P, _P],
                        _I),
    "hcw_decode_cache_bytes": ([_P, _I, _I, _I, _I, _I], _SZ),
    "hcw_block_workspace_bytes": ([_I, _I, _I, _I, _I, _I], _SZ),
    "hcw_block_step": ([_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _SZ, _P], _I),
    "hcw_gemm_workspace_bytes": ([_I, _I, _I], _SZ),
    "hcw_gemm_bf16": ([_I, _I, _I, _P, _I, _P, _I, _P, _P, _SZ, _P], _I),
    "hcw_gemm_bf16_batched": ([_I, _I, _I, _P, ctypes.c_longlong, _P, ctypes.c_longlong, _P, _I,
                               _P], _I),
    "hcw_set_stack_kernels": ([_I], _I),
    "hcw_set_decode_kernel": ([_I], _I),
    "hcw_stack_kernels_used": ([_I, _I, _I, _I], _I),
    "hcw_sync_status": ([_P], _I),
    "hcw_selftest_wait": ([_LL, _P], _I),
}

EXPORTED = tuple(_SIGNATURES)


class HcwError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s failed: %s (%d)" % (what, status_string(status), status))


def lib() -> ctypes.CDLL:
    """Load libhcw.so (built in-tree by build()); raise if it is missing."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    "libhcw.so not found at %s: run __graft_entry__.build() (or "
                    "python -m paper_2609_18145_gb300._build) first" % LIB_PATH)
            L = ctypes.CDLL(LIB_PATH)
            for name, (args, res) in _SIGNATURES.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = res
            _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().hcw_status_string(status).decode()


def _check(rc: int, what: str):
    if rc != HCW_OK:
        raise HcwError(rc, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return HCW_BF16
    if t.dtype == torch.float32:
        return HCW_F32
    raise TypeError("activations must be bfloat16 or float32, got %s" % t.dtype)


def _dev(*ts):
    for t in ts:
        if t is None:
            continue
        if not t.is_cuda:
            raise ValueError("all tensors must be CUDA tensors")
        if not t.is_contiguous():
            raise ValueError("all tensors must be contiguous")


def hcw_version() -> int:
    return lib().hcw_version()


def hcw_partner_table(layer: int, n: int, flags: int = 0, dim_override: int = -1):
    """Host partner table: list of n ints (-1 where the position does not receive)."""
    buf = (ctypes.c_int * n)()
    _check(lib().hcw_partner_table(layer, dim_override, n, flags, buf), "hcw_partner_table")
    return list(buf)


def hcw_partner_table_device(layer: int, n: int, flags: int = 0, dim_override: int = -1,
                             device=None, stream=None) -> torch.Tensor:
    out = torch.empty(n, dtype=torch.int32, device=device or "cuda")
    _check(lib().hcw_partner_table_device(layer, dim_override, n, flags, _ptr(out),
                                          _stream(stream)), "hcw_partner_table_device")
    return out


def hcw_layer_fwd(x, W_self, W_nbr, bias=None, layer: int = 0, dim_override: int = -1,
                  flags: int = 0, y=None, z_save=None, want_z: bool = False, stream=None):
    """One layer forward; returns y (and z_save if want_z or given)."""
    _dev(x, W_self, W_nbr, bias, y, z_save)
    B, n, d = x.shape
    if y is None:
        y = torch.empty_like(x)
    if want_z and z_save is None:
        z_save = torch.empty_like(x)
    _check(lib().hcw_layer_fwd(_ptr(x), _ptr(W_self), _ptr(W_nbr), _ptr(bias), layer,
                               dim_override, B, n, d, _dtype_code(x), flags, _ptr(y),
                               _ptr(z_save), _stream(stream)), "hcw_layer_fwd")
    return (y, z_save) if z_save is not None else y


def hcw_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int) -> int:
    return int(lib().hcw_workspace_bytes(B, n, d, dtype, flags))


def hcw_stack_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int, L: int) -> int:
    return int(lib().hcw_stack_workspace_bytes(B, n, d, dtype, flags, L))


def _workspace(nbytes, device, workspace):
    if workspace is not None:
        return workspace
    return torch.empty(max(nbytes, 1), dtype=torch.uint8, device=device)


def hcw_layer_bwd(x, z_save, dy, W_self, W_nbr, layer: int = 0, dim_override: int = -1,
                  flags: int = 0, dx=None, dW_self=None, dW_nbr=None, dbias=None,
                  want_dbias: bool = True, workspace=None, stream=None):
    """One layer backward; returns (dx, dW_self, dW_nbr, dbias)."""
    _dev(x, z_save, dy, W_self, W_nbr, dx, dW_self, dW_nbr, dbias, workspace)
    B, n, d = x.shape
    dt = _dtype_code(x)
    f32 = dict(dtype=torch.float32, device=x.device)
    dx = torch.empty_like(x) if dx is None else dx
    dW_self = torch.empty(d, d, **f32) if dW_self is None else dW_self
    dW_nbr = torch.empty(d, d, **f32) if dW_nbr is None else dW_nbr
    if dbias is None and want_dbias:
        dbias = torch.empty(d, **f32)
    need = hcw_workspace_bytes(B, n, d, dt, flags)
    ws = _workspace(need, x.device, workspace)
    _check(lib().hcw_layer_bwd(_ptr(x), _ptr(z_save), _ptr(dy), _ptr(W_self), _ptr(W_nbr),
                               layer, dim_override, B, n, d, dt, flags, _ptr(dx),
                               _ptr(dW_self), _ptr(dW_nbr), _ptr(dbias), _ptr(ws),
                               ws.numel(), _stream(stream)), "hcw_layer_bwd")
    return dx, dW_self, dW_nbr, dbias


def hcw_layer_bwd_data(dz, dy, W_self, W_nbr, layer: int = 0, dim_override: int = -1,
                       flags: int = 0, dx=None, stream=None):
    """Input gradient of one layer from dz = dy * act'(z); returns dx."""
    _dev(dz, dy, W_self, W_nbr, dx)
    B, n, d = dz.shape
    dx = torch.empty_like(dz) if dx is None else dx
    _check(lib().hcw_layer_bwd_data(_ptr(dz), _ptr(dy), _ptr(W_self), _ptr(W_nbr), layer,
                                    dim_override, B, n, d, _dtype_code(dz), flags, _ptr(dx),
                                    _stream(stream)), "hcw_layer_bwd_data")
    return dx


def hcw_layer_bwd_weight_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int) -> int:
    return int(lib().hcw_layer_bwd_weight_workspace_bytes(B, n, d, dtype, flags))


def hcw_layer_bwd_weight(x, dz, layer: int = 0, dim_override: int = -1, flags: int = 0,
                         dW_self=None, dW_nbr=None, dbias=None, want_dbias: bool = True,
                         workspace=None, stream=None):
    """Weight gradients of one layer; returns (dW_self, dW_nbr, dbias)."""
    _dev(x, dz, dW_self, dW_nbr, dbias, workspace)
    B, n, d = x.shape
    dt = _dtype_code(x)
    f32 = dict(dtype=torch.float32, device=x.device)
    dW_self = torch.empty(d, d, **f32) if dW_self is None else dW_self
    dW_nbr = torch.empty(d, d, **f32) if dW_nbr is None else dW_nbr
    if dbias is None and want_dbias:
        dbias = torch.empty(d, **f32)
    ws = _workspace(hcw_layer_bwd_weight_workspace_bytes(B, n, d, dt, flags), x.device,
                    workspace)
    _check(lib().hcw_layer_bwd_weight(_ptr(x), _ptr(dz), layer, dim_override, B, n, d, dt, flags,
                                      _ptr(dW_self), _ptr(dW_nbr), _ptr(dbias), _ptr(ws),
                                      ws.numel(), _stream(stream)), "hcw_layer_bwd_weight")
    return dW_self, dW_nbr, dbias


def hcw_decode_cache_bytes(L: int, B: int, n: int, d: int, dims=None, layer0: int = 0) -> int:
    arr = None if dims is None else _dims_array(dims, L)
    return int(lib().hcw_decode_cache_bytes(None if arr is None else ctypes.cast(arr, _P), layer0,
                                            L, B, n, d))


def hcw_decode_step(x_t, W_self, W_nbr, bias, t: int, n: int, cache, flags: int,
                    dims=None, layer0: int = 0, y=None, stream=None):
    """One decode step at position t (Sec. 6): x_t [B, d] bf16 in, returns y_t
    [B, d]; cache is the rings tensor of hcw_decode_cache_bytes (updated)."""
    _dev(x_t, W_self, W_nbr, bias, cache, y)
    B, d = x_t.shape
    L = W_self.shape[0]
    y = torch.empty_like(x_t) if y is None else y
    arr = None if dims is None else _dims_array(dims, L)
    _check(lib().hcw_decode_step(_ptr(x_t), _ptr(W_self), _ptr(W_nbr), _ptr(bias),
                                 None if arr is None else ctypes.cast(arr, _P), layer0, L, t, B,
                                 n, d, flags, _ptr(cache), _ptr(y), _stream(stream)),
           "hcw_decode_step")
    return y


BLOCK_FIELDS = ("E", "P", "ln1_g", "ln1_b", "W_self", "W_nbr", "ln2_g", "ln2_b", "W1", "b1",
                "W2", "b2", "lnf_g", "lnf_b", "Wh", "bh")


class _BlockPtrs(ctypes.Structure):
    """hcw_block_params / hcw_block_grads: sixteen device pointers in BLOCK_FIELDS order."""
    _fields_ = [(f, ctypes.c_void_p) for f in BLOCK_FIELDS]


def hcw_block_workspace_bytes(B: int, n: int, d: int, h: int, V: int, L: int) -> int:
    return int(lib().hcw_block_workspace_bytes(B, n, d, h, V, L))


def hcw_block_step(ids, params: dict, grads: dict | None = None, loss=None, workspace=None,
                   stream=None):
    """One training step of the character-LM block (forward, loss, backward).
    ids [B, n + 1] int32; params: BLOCK_FIELDS -> device tensors (bf16 tables
    and maps, fp32 LayerNorm parameters and biases).  Returns (loss [1] fp32,
    grads: BLOCK_FIELDS -> fp32 tensors of the parameters' shapes)."""
    _dev(ids, loss, workspace, *params.values())
    B, n1 = ids.shape
    n = n1 - 1
    V, d = params["E"].shape
    L, h = params["W1"].shape[0], params["W1"].shape[1]
    dev = ids.device
    if grads is None:
        grads = {f: torch.empty(tuple(params[f].shape), dtype=torch.float32, device=dev)
                 for f in BLOCK_FIELDS}
    loss = torch.empty(1, dtype=torch.float32, device=dev) if loss is None else loss
    ws = _workspace(hcw_block_workspace_bytes(B, n, d, h, V, L), dev, workspace)
    P = _BlockPtrs(*[params[f].data_ptr() for f in BLOCK_FIELDS])
    G = _BlockPtrs(*[grads[f].data_ptr() for f in BLOCK_FIELDS])
    _check(lib().hcw_block_step(_ptr(ids), ctypes.byref(P), ctypes.byref(G), B, n, d, h, V, L,
                                _ptr(loss), _ptr(ws), ws.numel(), _stream(stream)),
           "hcw_block_step")
    return loss, grads


def hcw_gemm_workspace_bytes(M: int, N: int, K: int) -> int:
    return int(lib().hcw_gemm_workspace_bytes(M, N, K))


def hcw_gemm_bf16(A, B, ta: bool = False, tb: bool = False, C=None, workspace=None,
                  split: bool = True, stream=None):
    """fp32 C = op(A) op(B) from bf16 A ([M, K], or [K, M] with ta) and B
    ([K, N], or [N, K] with tb).  split=False passes no workspace (no K
    split).  Returns C [M, N]."""
    _dev(A, B, C, workspace)
    if A.dtype != torch.bfloat16 or B.dtype != torch.bfloat16 or A.dim() != 2 or B.dim() != 2:
        raise ValueError("hcw_gemm_bf16: A and B must be 2-D bf16 tensors")
    M, K = (A.shape[1], A.shape[0]) if ta else (A.shape[0], A.shape[1])
    Kb, N = (B.shape[1], B.shape[0]) if tb else (B.shape[0], B.shape[1])
    if Kb != K:
        raise ValueError("hcw_gemm_bf16: inner sizes differ (%d, %d)" % (K, Kb))
    C = torch.empty(M, N, dtype=torch.float32, device=A.device) if C is None else C
    if split:
        ws = _workspace(hcw_gemm_workspace_bytes(M, N, K), A.device, workspace)
        wp, wn = _ptr(ws), ws.numel()
    else:
        wp, wn = None, 0
    _check(lib().hcw_gemm_bf16(M, N, K, _ptr(A), int(bool(ta)), _ptr(B), int(bool(tb)), _ptr(C),
                               wp, wn, _stream(stream)), "hcw_gemm_bf16")
    return C


def hcw_gemm_bf16_batched(A, B, C=None, stream=None):
    """fp32 C[b] = A[b]^T B[b] from bf16 A [batch, K, M] and B [batch, K, N]
    (each product contracted over its rows, whole K per output tile).  The
    batch dimension may have any stride (in elements); the rows are
    contiguous.  Returns C [batch, M, N]."""
    _dev(C)
    if not (A.is_cuda and B.is_cuda):
        raise ValueError("all tensors must be CUDA tensors")
    if A.dtype != torch.bfloat16 or B.dtype != torch.bfloat16 or A.dim() != 3 or B.dim() != 3:
        raise ValueError("hcw_gemm_bf16_batched: A and B must be 3-D bf16 tensors")
    batch, K, M = A.shape
    if B.shape[0] != batch or B.shape[1] != K:
        raise ValueError("hcw_gemm_bf16_batched: A %s and B %s do not match"
                         % (tuple(A.shape), tuple(B.shape)))
    N = B.shape[2]
    if A.stride(2) != 1 or A.stride(1) != M or B.stride(2) != 1 or B.stride(1) != N:
        raise ValueError("hcw_gemm_bf16_batched: each product's rows must be contiguous")
    C = torch.empty(batch, M, N, dtype=torch.float32, device=A.device) if C is None else C
    _check(lib().hcw_gemm_bf16_batched(M, N, K, _ptr(A), A.stride(0), _ptr(B), B.stride(0),
                                       _ptr(C), batch, _stream(stream)), "hcw_gemm_bf16_batched")
    return C


def hcw_set_decode_kernel(mode: int) -> int:
    """Select the contraction of hcw_decode_step (HCW_DECODE_WARP_MMA or
    HCW_DECODE_TCGEN05) for this process; returns the previous mode."""
    prev = int(lib().hcw_set_decode_kernel(int(mode)))
    if prev < 0:
        raise ValueError("hcw_set_decode_kernel: unknown mode %r" % (mode,))
    return prev


def hcw_set_stack_kernels(mode: int) -> int:
    """Select the bf16 stacked-launch kernels (HCW_STACK_AUTO, _RESIDENT or
    _STREAMING) for this process; returns the previous mode."""
    prev = int(lib().hcw_set_stack_kernels(int(mode)))
    if prev < 0:
        raise ValueError("hcw_set_stack_kernels: unknown mode %r" % (mode,))
    return prev


def hcw_stack_kernels_used(B: int, n: int, d: int, dtype: int = HCW_BF16) -> int:
    """HCW_STACK_RESIDENT or HCW_STACK_STREAMING: the family a bf16 stack of
    these sizes runs on under the current setting."""
    r = int(lib().hcw_stack_kernels_used(B, n, d, dtype))
    if r < 0:
        raise ValueError("hcw_stack_kernels_used: invalid sizes")
    return r


def hcw_launch_count() -> int:
    """Kernels launched by libhcw in this process so far."""
    return int(lib().hcw_launch_count())


def hcw_stack_fwd_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int, L: int) -> int:
    return int(lib().hcw_stack_fwd_workspace_bytes(B, n, d, dtype, flags, L))


def _dims_array(dims, L):
    """A layer schedule as a C int array of L dimensions (kept alive by the caller)."""
    vals = [int(v) for v in dims]
    if len(vals) != L:
        raise ValueError("dims needs one cube dimension per layer (%d), got %d" % (L, len(vals)))
    return (ctypes.c_int * L)(*vals)


def hcw_stack_fwd(x, W_self, W_nbr, bias=None, layer0: int = 0, dim_override: int = -1,
                  flags: int = 0, y=None, acts=None, masks=None, want_masks: bool = None,
                  workspace=None, stream=None, dims=None):
    """Stack forward over L = W_self.shape[0] layers; returns (y, acts, masks).
    masks (ReLU only) are int32 words [L, B, n, ceil(d/32)], bit o%32 of word
    o/32 = (z > 0); allocated when the stack uses ReLU unless want_masks=False.
    dims (a sequence of L cube dimensions) calls hcw_stack_fwd_dims instead;
    layer0 and dim_override are then unused."""
    _dev(x, W_self, W_nbr, bias, y, acts, masks, workspace)
    B, n, d = x.shape
    L = W_self.shape[0]
    dt = _dtype_code(x)
    y = torch.empty_like(x) if y is None else y
    if acts is None and L > 1:
        acts = torch.empty((L - 1, B, n, d), dtype=x.dtype, device=x.device)
    if want_masks is None:
        want_masks = bool(flags & HCW_ACT_RELU)
    if masks is None and want_masks:
        masks = torch.empty((L, B, n, (d + 31) // 32), dtype=torch.int32, device=x.device)
    ws = _workspace(hcw_stack_fwd_workspace_bytes(B, n, d, dt, flags, L), x.device, workspace)
    if dims is not None:
        arr = _dims_array(dims, L)
        _check(lib().hcw_stack_fwd_dims(_ptr(x), _ptr(W_self), _ptr(W_nbr), _ptr(bias),
                                        ctypes.cast(arr, _P), L, B, n, d, dt, flags, _ptr(y),
                                        _ptr(acts), _ptr(masks), _ptr(ws), ws.numel(),
                                        _stream(stream)), "hcw_stack_fwd_dims")
        return y, acts, masks
    _check(lib().hcw_stack_fwd(_ptr(x), _ptr(W_self), _ptr(W_nbr), _ptr(bias), layer0, L,
                               dim_override, B, n, d, dt, flags, _ptr(y), _ptr(acts),
                               _ptr(masks), _ptr(ws), ws.numel(), _stream(stream)),
           "hcw_stack_fwd")
    return y, acts, masks


def hcw_stack_fwd_dims(x, W_self, W_nbr, bias, dims, flags: int = 0, **kw):
    """hcw_stack_fwd with layer l on cube dimension dims[l]."""
    return hcw_stack_fwd(x, W_self, W_nbr, bias, flags=flags, dims=dims, **kw)


def hcw_stack_bwd(x, acts, masks, dy, W_self, W_nbr, layer0: int = 0, dim_override: int = -1,
                  flags: int = 0, dx=None, dW_self=None, dW_nbr=None, dbias=None,
                  want_dbias: bool = True, workspace=None, stream=None, dims=None):
    """Stack backward; returns (dx, dW_self[L], dW_nbr[L], dbias[L]).  dims as
    for hcw_stack_fwd (calls hcw_stack_bwd_dims)."""
    _dev(x, acts, masks, dy, W_self, W_nbr, dx, dW_self, dW_nbr, dbias, workspace)
    B, n, d = x.shape
    L = W_self.shape[0]
    dt = _dtype_code(x)
    f32 = dict(dtype=torch.float32, device=x.device)
    dx = torch.empty_like(x) if dx is None else dx
    dW_self = torch.empty(L, d, d, **f32) if dW_self is None else dW_self
    dW_nbr = torch.empty(L, d, d, **f32) if dW_nbr is None else dW_nbr
    if dbias is None and want_dbias:
        dbias = torch.empty(L, d, **f32)
    need = hcw_stack_workspace_bytes(B, n, d, dt, flags, L)
    ws = _workspace(need, x.device, workspace)
    if dims is not None:
        arr = _dims_array(dims, L)
        _check(lib().hcw_stack_bwd_dims(_ptr(x), _ptr(acts), _ptr(masks), _ptr(dy),
                                        _ptr(W_self), _ptr(W_nbr), ctypes.cast(arr, _P), L, B,
                                        n, d, dt, flags, _ptr(dx), _ptr(dW_self), _ptr(dW_nbr),
                                        _ptr(dbias), _ptr(ws), ws.numel(), _stream(stream)),
               "hcw_stack_bwd_dims")
        return dx, dW_self, dW_nbr, dbias
    _check(lib().hcw_stack_bwd(_ptr(x), _ptr(acts), _ptr(masks), _ptr(dy), _ptr(W_self),
                               _ptr(W_nbr), layer0, L, dim_override, B, n, d, dt, flags,
                               _ptr(dx), _ptr(dW_self), _ptr(dW_nbr), _ptr(dbias), _ptr(ws),
                               ws.numel(), _stream(stream)), "hcw_stack_bwd")
    return dx, dW_self, dW_nbr, dbias


def hcw_stack_train_step_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int,
                                         L: int) -> int:
    return int(lib().hcw_stack_train_step_workspace_bytes(B, n, d, dtype, flags, L))


def hcw_stack_train_step(x, W_self, W_nbr, bias, dy, layer0: int = 0, dim_override: int = -1,
                         flags: int = 0, y=None, acts=None, masks=None, dx=None, dW_self=None,
                         dW_nbr=None, dbias=None, want_dbias: bool = True,
                         want_dw: bool = True, workspace=None, stream=None, dims=None):
    """Forward and backward of a stack in one call; returns (y, acts, masks,
    dx, dW_self[L], dW_nbr[L], dbias[L]).  want_dw=False: the forward and the
    input gradient only (the weight-gradient outputs are None).  dims (a
    sequence of L layer links, as for hcw_stack_fwd) calls
    hcw_stack_train_step_dims instead; layer0 and dim_override are then
    ignored."""
    _dev(x, W_self, W_nbr, bias, dy, y, acts, masks, dx, dW_self, dW_nbr, dbias, workspace)
    B, n, d = x.shape
    L = W_self.shape[0]
    dt = _dtype_code(x)
    f32 = dict(dtype=torch.float32, device=x.device)
    y = torch.empty_like(x) if y is None else y
    if acts is None and L > 1:
        acts = torch.empty((L - 1, B, n, d), dtype=x.dtype, device=x.device)
    if masks is None and flags & HCW_ACT_RELU:
        masks = torch.empty((L, B, n, (d + 31) // 32), dtype=torch.int32, device=x.device)
    dx = torch.empty_like(x) if dx is None else dx
    if want_dw:
        dW_self = torch.empty(L, d, d, **f32) if dW_self is None else dW_self
        dW_nbr = torch.empty(L, d, d, **f32) if dW_nbr is None else dW_nbr
        if dbias is None and want_dbias:
            dbias = torch.empty(L, d, **f32)
    ws = _workspace(hcw_stack_train_step_workspace_bytes(B, n, d, dt, flags, L), x.device,
                    workspace)
    if dims is not None:
        arr = _dims_array(dims, L)
        _check(lib().hcw_stack_train_step_dims(_ptr(x), _ptr(W_self), _ptr(W_nbr), _ptr(bias),
                                               _ptr(dy), arr, L, B, n, d, dt, flags, _ptr(y),
                                               _ptr(acts), _ptr(masks), _ptr(dx),
                                               _ptr(dW_self), _ptr(dW_nbr), _ptr(dbias),
                                               _ptr(ws), ws.numel(), _stream(stream)),
               "hcw_stack_train_step_dims")
        return y, acts, masks, dx, dW_self, dW_nbr, dbias
    _check(lib().hcw_stack_train_step(_ptr(x), _ptr(W_self), _ptr(W_nbr), _ptr(bias), _ptr(dy),
                                      layer0, L, dim_override, B, n, d, dt, flags, _ptr(y),
                                      _ptr(acts), _ptr(masks), _ptr(dx),
                                      _ptr(dW_self), _ptr(dW_nbr), _ptr(dbias), _ptr(ws),
                                      ws.numel(), _stream(stream)), "hcw_stack_train_step")
    return y, acts, masks, dx, dW_self, dW_nbr, dbias


def hcw_stack_bwd_dims(x, acts, masks, dy, W_self, W_nbr, dims, flags: int = 0, **kw):
    """hcw_stack_bwd of a stack run with hcw_stack_fwd_dims(dims)."""
    return hcw_stack_bwd(x, acts, masks, dy, W_self, W_nbr, flags=flags, dims=dims, **kw)


def hcw_stack_bwd_data_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int,
                                       L: int) -> int:
    return int(lib().hcw_stack_bwd_data_workspace_bytes(B, n, d, dtype, flags, L))


def hcw_stack_bwd_weight_workspace_bytes(B: int, n: int, d: int, dtype: int, flags: int,
                                         L: int) -> int:
    return int(lib().hcw_stack_bwd_weight_workspace_bytes(B, n, d, dtype, flags, L))


def hcw_stack_bwd_data(masks, dy, W_self, W_nbr, layer0: int = 0, dim_override: int = -1,
                       flags: int = 0, dx=None, dz=None, workspace=None, stream=None):
    """Input gradients through the stack; returns (dx, dz[L])."""
    _dev(masks, dy, W_self, W_nbr, dx, dz, workspace)
    B, n, d = dy.shape
    L = W_self.shape[0]
    dt = _dtype_code(dy)
    dx = torch.empty_like(dy) if dx is None else dx
    dz = torch.empty((L, B, n, d), dtype=dy.dtype, device=dy.device) if dz is None else dz
    need = hcw_stack_bwd_data_workspace_bytes(B, n, d, dt, flags, L)
    ws = _workspace(need, dy.device, workspace)
    _check(lib().hcw_stack_bwd_data(_ptr(masks), _ptr(dy), _ptr(W_self), _ptr(W_nbr), layer0, L,
                                    dim_override, B, n, d, dt, flags, _ptr(dx), _ptr(dz),
                                    _ptr(ws), ws.numel(), _stream(stream)), "hcw_stack_bwd_data")
    return dx, dz


def hcw_stack_bwd_weight(x, acts, dz, layer0: int = 0, dim_override: int = -1, flags: int = 0,
                         dW_self=None, dW_nbr=None, dbias=None, want_dbias: bool = True,
                         workspace=None, stream=None, dims=None):
    """Weight gradients of every layer from its input and dz; returns
    (dW_self[L], dW_nbr[L], dbias[L] or None).  dims (L layer links) calls
    hcw_stack_bwd_weight_dims instead."""
    _dev(x, acts, dz, dW_self, dW_nbr, dbias, workspace)
    B, n, d = x.shape
    L = dz.shape[0]
    dt = _dtype_code(x)
    f32 = dict(dtype=torch.float32, device=x.device)
    dW_self = torch.empty(L, d, d, **f32) if dW_self is None else dW_self
    dW_nbr = torch.empty(L, d, d, **f32) if dW_nbr is None else dW_nbr
    if dbias is None and want_dbias:
        dbias = torch.empty(L, d, **f32)
    need = hcw_stack_bwd_weight_workspace_bytes(B, n, d, dt, flags, L)
    ws = _workspace(need, x.device, workspace)
    if dims is not None:
        _check(lib().hcw_stack_bwd_weight_dims(_ptr(x), _ptr(acts), _ptr(dz), _dims_array(dims, L),
                                               L, B, n, d, dt, flags, _ptr(dW_self),
                                               _ptr(dW_nbr), _ptr(dbias), _ptr(ws), ws.numel(),
                                               _stream(stream)), "hcw_stack_bwd_weight_dims")
        return dW_self, dW_nbr, dbias
    _check(lib().hcw_stack_bwd_weight(_ptr(x), _ptr(acts), _ptr(dz), layer0, L, dim_override,
                                      B, n, d, dt, flags, _ptr(dW_self), _ptr(dW_nbr),
                                      _ptr(dbias), _ptr(ws), ws.numel(), _stream(stream)),
           "hcw_stack_bwd_weight")
    return dW_self, dW_nbr, dbias


def hcw_sync_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device error status."""
    return int(lib().hcw_sync_status(_stream(stream)))


def hcw_selftest_wait(timeout_ns: int, stream=None):
    _check(lib().hcw_selftest_wait(int(timeout_ns), _stream(stream)), "hcw_selftest_wait")
