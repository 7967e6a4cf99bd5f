"""CPU ORACLE for the PARD speculative decode step -- test infrastructure.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg (and its ``--impl reference`` arm) may import this package.  It is a
plain, slow, obviously-correct fp32 restatement of the paper's method and
shares no code with the CUDA path:

* ``forward.c``  -- Llama-style decoder forward (fp32, fixed summation order)
* ``philox.py``  -- Philox4x32-10 from its published definition
* ``pard.py``    -- the PARD decode step: parallel draft with mask tokens
  (Eq. 6), target verification (Section 2.2), greedy and speculative-sampling
  acceptance, KV commit and rollback, and autoregressive greedy decoding
  (Eq. 2) as the lossless reference.

Parity status: every function is pinned by ``tests/test_oracle_*.py``
(closed forms, invariants, library routines, brute force on tiny inputs);
the logit values of a whole random-init model have no printed value in the
paper and are pinned only through those pieces.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None

T_PER_LAYER = 9
LAYER_ORDER = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")


class OCfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d", ctypes.c_int32), ("hq", ctypes.c_int32),
                ("hkv", ctypes.c_int32), ("hd", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("theta", ctypes.c_float), ("eps", ctypes.c_float)]


class OWeights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p), ("layers", ctypes.POINTER(ctypes.c_void_p))]


def _build_lib() -> str:
    src = os.path.join(_HERE, "forward.c")
    out = os.path.join(_HERE, "_oracle_forward.so")
    if os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    subprocess.check_call(["gcc", "-O2", "-std=c99", "-fopenmp", "-fPIC", "-shared",
                           "-ffp-contract=off", "-fno-fast-math", src, "-o", tmp, "-lm"])
    os.replace(tmp, out)
    return out


def build() -> None:
    """Compile the oracle's C part (idempotent)."""
    lib()


def lib():
    global _LIB
    if _LIB is None:
        L = ctypes.CDLL(_build_lib())
        fp, i32, vp = ctypes.c_float, ctypes.c_int32, ctypes.c_void_p
        L.oracle_forward.argtypes = [ctypes.POINTER(OCfg), ctypes.POINTER(OWeights), vp, vp, i32,
                                     vp, i32, vp, vp, i32, vp, vp, i32]
        L.oracle_forward.restype = ctypes.c_int
        L.oracle_matmul.argtypes = [vp, i32, i32, vp, i32, vp]
        L.oracle_matmul_cols.argtypes = [vp, i32, i32, vp, vp, i32, vp]
        L.oracle_rmsnorm.argtypes = [vp, vp, i32, fp, vp]
        L.oracle_rope.argtypes = [vp, i32, i32, fp]
        L.oracle_attend.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp, vp]
        _LIB = L
    return _LIB


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


# --------------------------------------------------------------------------
# Thin numpy wrappers around the C primitives
# --------------------------------------------------------------------------
def matmul(x: np.ndarray, w_bits: np.ndarray) -> np.ndarray:
    """x fp32 [m, K] times bf16 W [N, K] transposed -> fp32 [m, N]."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    w_bits = np.ascontiguousarray(w_bits, dtype=np.uint16)
    m, K = x.shape
    N = w_bits.shape[0]
    assert w_bits.shape[1] == K
    y = np.empty((m, N), dtype=np.float32)
    lib().oracle_matmul(_ptr(x), m, K, _ptr(w_bits), N, _ptr(y))
    return y


def matmul_cols(x: np.ndarray, w_bits: np.ndarray, cols) -> np.ndarray:
    """Only output columns ``cols`` of matmul(x, w_bits)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    cols = np.ascontiguousarray(cols, dtype=np.int32)
    m, K = x.shape
    y = np.empty((m, len(cols)), dtype=np.float32)
    lib().oracle_matmul_cols(_ptr(x), m, K, _ptr(np.ascontiguousarray(w_bits)), _ptr(cols),
                             len(cols), _ptr(y))
    return y


def rmsnorm(x: np.ndarray, g_bits: np.ndarray, eps: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty_like(x)
    d = x.shape[-1]
    g_bits = np.ascontiguousarray(g_bits, dtype=np.uint16)
    for r in range(x.reshape(-1, d).shape[0]):
        lib().oracle_rmsnorm(_ptr(x.reshape(-1, d)[r]), _ptr(g_bits), d, eps,
                             out.reshape(-1, d)[r].ctypes.data)
    return out


def rope(v: np.ndarray, pos: int, theta: float) -> np.ndarray:
    """RoPE of one head vector (rotate-half pairs)."""
    out = np.array(v, dtype=np.float32, copy=True)
    lib().oracle_rope(_ptr(out), out.shape[0], int(pos), theta)
    return out


def attend(q: np.ndarray, kc: np.ndarray, vc: np.ndarray, kvh: int, pos: int) -> np.ndarray:
    """One query over cache positions 0..pos; kc/vc are [max_pos, hkv, hd]."""
    q = np.ascontiguousarray(q, dtype=np.float32)
    kc = np.ascontiguousarray(kc, dtype=np.float32)
    vc = np.ascontiguousarray(vc, dtype=np.float32)
    hkv, hd = kc.shape[1], kc.shape[2]
    scratch = np.empty(kc.shape[0], dtype=np.float32)
    out = np.empty(hd, dtype=np.float32)
    lib().oracle_attend(_ptr(q), _ptr(kc), _ptr(vc), hkv, hd, kvh, int(pos), _ptr(scratch), _ptr(out))
    return out


from .pard import OracleModel, OracleDecoder, ar_greedy, accept_greedy, accept_sampling  # noqa: E402,F401
