"""fp64 CPU oracle for ragged causal GQA prefill attention (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path never does: the CUDA
library and this oracle share no code.  The arithmetic lives in ``oracle.c``
(plain C, one output row at a time, explicit two-pass softmax); this module
only compiles it with gcc and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
# A prebuilt variant of the library, loaded instead of building oracle.c: the
# mutation tests point it at copies of oracle.c with a mistake planted in them.
_OVERRIDE = os.environ.get("OPATTN_ORACLE_LIBRARY")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it (gcc, no -march flags)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
                        "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            if _OVERRIDE:
                lib = ctypes.CDLL(_OVERRIDE)
            else:
                build()
                lib = ctypes.CDLL(_LIB)
            p = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_attention_rows.argtypes = [p, p, p, p, p, i32, i32, i32, i32, f64,
                                                  p, p, i64, p, p, i32]
            lib.oracle_attention_rows.restype = ctypes.c_int
            lib.oracle_attention.argtypes = [p, p, p, p, p, i32, i32, i32, i32, f64, p, p, i32]
            lib.oracle_attention.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _bits(x) -> np.ndarray:
    """bf16 bit patterns as a contiguous uint16 numpy array (torch or numpy input)."""
    if hasattr(x, "view") and hasattr(x, "dtype") and str(x.dtype) == "torch.bfloat16":
        import torch
        x = x.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)
    a = np.ascontiguousarray(x)
    if a.dtype != np.uint16:
        raise TypeError("oracle inputs are bf16 bit patterns (uint16) or bf16 torch tensors")
    return a


def default_threads() -> int:
    return os.cpu_count() or 1


def attention(q, k, v, cu_q, cu_k, Hq: int, Hkv: int, d: int, scale: float,
              n_threads: int | None = None):
    """All rows.  Returns (o [total_q, Hq, d] float64, lse [total_q, Hq] float64)."""
    lib = _load()
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    cq = np.ascontiguousarray(cu_q, dtype=np.int32)
    ck = np.ascontiguousarray(cu_k, dtype=np.int32)
    n_seq = len(cq) - 1
    total_q = int(cq[-1])
    o = np.zeros((total_q, Hq, d), dtype=np.float64)
    lse = np.zeros((total_q, Hq), dtype=np.float64)
    rc = lib.oracle_attention(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(cq), _ptr(ck), n_seq,
                              Hq, Hkv, d, float(scale), _ptr(o), _ptr(lse),
                              n_threads or default_threads())
    if rc != 0:
        raise ValueError("oracle_attention rejected its arguments")
    return o, lse


def attention_rows(q, k, v, cu_q, cu_k, Hq: int, Hkv: int, d: int, scale: float,
                   tokens, heads, n_threads: int | None = None):
    """Selected rows (tokens[r], heads[r]).  Returns (o [n, d], lse [n]) float64."""
    lib = _load()
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    cq = np.ascontiguousarray(cu_q, dtype=np.int32)
    ck = np.ascontiguousarray(cu_k, dtype=np.int32)
    t = np.ascontiguousarray(tokens, dtype=np.int64)
    h = np.ascontiguousarray(heads, dtype=np.int32)
    n = len(t)
    o = np.zeros((n, d), dtype=np.float64)
    lse = np.zeros((n,), dtype=np.float64)
    rc = lib.oracle_attention_rows(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(cq), _ptr(ck),
                                   len(cq) - 1, Hq, Hkv, d, float(scale), _ptr(t), _ptr(h),
                                   n, _ptr(o), _ptr(lse), n_threads or default_threads())
    if rc != 0:
        raise ValueError("oracle_attention_rows rejected its arguments")
    return o, lse
