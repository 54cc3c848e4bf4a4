"""ctypes front end of the fp64 CPU oracle (``oracle.c``).

TEST INFRASTRUCTURE, NOT PRODUCT CODE: only the test suite, the smoke check
and the CPU-baseline leg of the benchmark import this module.  The CUDA path
never does, and this module imports nothing from the CUDA path.

Every array argument is a float64 numpy array (converted here if needed);
layouts follow ``oracle.c``: activations [B, n, d], weights [d_out, d_in]
acting on column vectors as in Eq. (1), stacks with a leading layer axis.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

CAUSAL = 1
RESIDUAL = 2
ACT_RELU = 4

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, OpenMP, no fast-math)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".%d.tmp" % os.getpid()
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            U = ctypes.c_uint
            lib.oracle_dim.argtypes = [I, I, I]
            lib.oracle_partner.argtypes = [I, I]
            lib.oracle_receives.argtypes = [I, I, U]
            lib.oracle_partner_table.argtypes = [I, I, I, U, P]
            lib.oracle_round_bf16.argtypes = [ctypes.c_double]
            lib.oracle_round_bf16.restype = ctypes.c_double
            lib.oracle_round_bf16_array.argtypes = [P, ctypes.c_longlong]
            lib.oracle_layer_fwd.argtypes = [P, P, P, P, I, I, I, I, I, U, I, P, P]
            lib.oracle_layer_bwd.argtypes = [P, P, P, P, P, I, I, I, I, I, U, I, P, P, P, P]
            lib.oracle_stack_fwd.argtypes = [P, P, P, P, P, I, I, I, I, I, I, U, I, P, P, P]
            lib.oracle_stack_bwd.argtypes = [P, P, P, P, P, P, I, I, I, I, I, I, U, I,
                                             P, P, P, P]
            _lib = lib
    return _lib


def _f64(a):
    if a is None:
        return None
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def dim(layer: int, dim_override: int, n: int) -> int:
    return int(_load().oracle_dim(layer, dim_override, n))


def partner(i: int, s: int) -> int:
    return int(_load().oracle_partner(i, s))


def receives(i: int, s: int, flags: int) -> int:
    return int(_load().oracle_receives(i, s, flags))


def partner_table(layer: int, dim_override: int, n: int, flags: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    rc = _load().oracle_partner_table(layer, dim_override, n, flags, _p(out))
    if rc != 0:
        raise ValueError("invalid layer/n")
    return out


def round_bf16(v):
    """Round each value to the nearest bfloat16 (ties to even)."""
    arr = np.array(v, dtype=np.float64, order="C", copy=True)
    _load().oracle_round_bf16_array(_p(arr), arr.size)
    return arr if arr.ndim else float(arr)


def layer_fwd(x, W_self, W_nbr, bias, layer, dim_override, flags, round_bf16=False,
              want_z=False):
    """One layer forward; returns y (and z if want_z)."""
    x = _f64(x)
    B, n, d = x.shape
    Ws, Wn, b = _f64(W_self), _f64(W_nbr), _f64(bias)
    y = np.empty_like(x)
    z = np.empty_like(x) if want_z else None
    rc = _load().oracle_layer_fwd(_p(x), _p(Ws), _p(Wn), _p(b), layer, dim_override,
                                  B, n, d, flags, int(round_bf16), _p(y), _p(z))
    if rc != 0:
        raise ValueError("oracle_layer_fwd rejected its arguments")
    return (y, z) if want_z else y


def layer_bwd(x, z, dy, W_self, W_nbr, layer, dim_override, flags, round_bf16=False):
    """One layer backward; returns (dx, dW_self, dW_nbr, dbias)."""
    x, dy = _f64(x), _f64(dy)
    z = _f64(z)
    B, n, d = x.shape
    Ws, Wn = _f64(W_self), _f64(W_nbr)
    dx = np.empty_like(x)
    dWs = np.empty((d, d))
    dWn = np.empty((d, d))
    db = np.empty(d)
    rc = _load().oracle_layer_bwd(_p(x), _p(z), _p(dy), _p(Ws), _p(Wn), layer,
                                  dim_override, B, n, d, flags, int(round_bf16),
                                  _p(dx), _p(dWs), _p(dWn), _p(db))
    if rc != 0:
        raise ValueError("oracle_layer_bwd rejected its arguments")
    return dx, dWs, dWn, db


def stack_fwd(x, W_self, W_nbr, bias, layer0, L, dim_override, flags, round_bf16=False,
              dims=None):
    """Stack forward; returns (y, acts[L], zs[L]) with acts[l] = input of layer l."""
    x = _f64(x)
    B, n, d = x.shape
    Ws, Wn, b = _f64(W_self), _f64(W_nbr), _f64(bias)
    dd = None if dims is None else np.ascontiguousarray(np.asarray(dims, dtype=np.int32))
    y = np.empty_like(x)
    acts = np.empty((L, B, n, d))
    zs = np.empty((L, B, n, d))
    rc = _load().oracle_stack_fwd(_p(x), _p(Ws), _p(Wn), _p(b), _p(dd), layer0, L,
                                  dim_override, B, n, d, flags, int(round_bf16),
                                  _p(y), _p(acts), _p(zs))
    if rc != 0:
        raise ValueError("oracle_stack_fwd rejected its arguments")
    return y, acts, zs


def stack_bwd(acts, zs, dy, W_self, W_nbr, layer0, L, dim_override, flags,
              round_bf16=False, dims=None):
    """Stack backward; returns (dx, dW_self[L], dW_nbr[L], dbias[L])."""
    acts, zs, dy = _f64(acts), _f64(zs), _f64(dy)
    _, B, n, d = acts.shape
    Ws, Wn = _f64(W_self), _f64(W_nbr)
    dd = None if dims is None else np.ascontiguousarray(np.asarray(dims, dtype=np.int32))
    dx = np.empty((B, n, d))
    dWs = np.empty((L, d, d))
    dWn = np.empty((L, d, d))
    db = np.empty((L, d))
    rc = _load().oracle_stack_bwd(_p(acts), _p(zs), _p(dy), _p(Ws), _p(Wn), _p(dd), layer0,
                                  L, dim_override, B, n, d, flags, int(round_bf16),
                                  _p(dx), _p(dWs), _p(dWn), _p(db))
    if rc != 0:
        raise ValueError("oracle_stack_bwd rejected its arguments")
    return dx, dWs, dWn, db
