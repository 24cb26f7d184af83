"""Python binding of libopattn (ragged causal GQA prefill and decode attention on GB300).

Argument marshalling only: every step of the computation runs in the CUDA
library behind the C ABI declared in ``include/opattn.h``.  PyTorch is used
for device memory and streams.  There is no fallback: if ``libopattn.so`` has
not been built, every entry point raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libopattn.so")

OPATTN_OK = 0
OPATTN_ERR_INVALID_ARG = 1
OPATTN_ERR_UNSUPPORTED = 2
OPATTN_ERR_MISALIGNED = 3
OPATTN_ERR_CUDA = 4
OPATTN_ERR_TIMEOUT = 5
OPATTN_ERR_CAPACITY = 6
OPATTN_FLAG_TEST_FORCE_TIMEOUT = 1
OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA = 2
OPATTN_NOALLOC_MAX_UNITS = 32768

UNIT_FIELDS = ("q_tok0", "n_tok", "k_row0", "Lk", "qlim0", "kvh", "n_tiles", "seq", "tile0", "part", "group", "chunk",
               "n_chunks")
DEC_UNIT_FIELDS = ("q_tok0", "nq", "k_row0", "Lk", "kvh", "tile0", "n_tiles", "part", "group", "chunk", "n_chunks",
                   "seq")
DEC_COLS = 32

_lock = threading.Lock()
_lib = None


class OpattnError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


def load():
    """Load libopattn.so (built by ``paper_2608_13499_gb300.build.build()``)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise ImportError(f"{LIB_PATH} is missing: build it with paper_2608_13499_gb300.build.build() "
                                  "(nvcc, sm_103a); there is no fallback implementation")
            lib = ctypes.CDLL(LIB_PATH)
            P, i32, i64, u32, f32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                     ctypes.c_float)
            lib.opattn_version.restype = i32
            lib.opattn_version.argtypes = []
            lib.opattn_status_string.restype = ctypes.c_char_p
            lib.opattn_status_string.argtypes = [i32]
            lib.opattn_prefill.restype = ctypes.c_int
            lib.opattn_prefill.argtypes = [P, P, P, P, P, P, P, i32, i32, i32, i32, f32, P]
            lib.opattn_prefill_noalloc.restype = ctypes.c_int
            lib.opattn_prefill_noalloc.argtypes = [P, P, P, P, P, P, P, i32, i32, i32, i32, f32, P]
            lib.opattn_prefill_checked.restype = ctypes.c_int
            lib.opattn_prefill_checked.argtypes = [P, P, P, P, P, P, P, i32, i32, i32, i32, f32, P, u32]
            lib.opattn_plan_create.restype = ctypes.c_int
            lib.opattn_plan_create.argtypes = [ctypes.POINTER(P), P, P, i32, i32, i32, i32, i32]
            lib.opattn_plan_run.restype = ctypes.c_int
            lib.opattn_plan_run.argtypes = [P, P, P, P, P, P, f32, P]
            lib.opattn_plan_run_checked.restype = ctypes.c_int
            lib.opattn_plan_run_checked.argtypes = [P, P, P, P, P, P, f32, P, u32]
            lib.opattn_plan_destroy.restype = ctypes.c_int
            lib.opattn_plan_destroy.argtypes = [P]
            lib.opattn_plan_info.restype = ctypes.c_int
            lib.opattn_plan_info.argtypes = [P, ctypes.POINTER(i64), ctypes.POINTER(i32)]
            lib.opattn_schedule.restype = ctypes.c_int
            lib.opattn_schedule.argtypes = [P, P, i32, i32, i32, i32, i32, P, i64, P,
                                            ctypes.POINTER(i64), ctypes.POINTER(i32)]
            lib.opattn_decode.restype = ctypes.c_int
            lib.opattn_decode.argtypes = [P, P, P, P, P, P, P, i32, i32, i32, i32, f32, P]
            lib.opattn_decode_checked.restype = ctypes.c_int
            lib.opattn_decode_checked.argtypes = [P, P, P, P, P, P, P, i32, i32, i32, i32, f32, P, u32]
            lib.opattn_decode_plan_create.restype = ctypes.c_int
            lib.opattn_decode_plan_create.argtypes = [ctypes.POINTER(P), P, P, i32, i32, i32, i32, i32]
            lib.opattn_decode_paged.restype = ctypes.c_int
            lib.opattn_decode_paged.argtypes = [P, P, P, P, i64, i32, i32, P, P, P, P, i32, i32, i32, i32, f32, P]
            lib.opattn_decode_paged_plan_create.restype = ctypes.c_int
            lib.opattn_decode_paged_plan_create.argtypes = [ctypes.POINTER(P), P, P, i32, i32, i32, i32, i32, i32,
                                                            i32]
            lib.opattn_prefill_paged.restype = ctypes.c_int
            lib.opattn_prefill_paged.argtypes = [P, P, P, P, i64, i32, i32, P, P, P, P, i32, i32, i32, i32, f32, P]
            lib.opattn_prefill_paged_plan_create.restype = ctypes.c_int
            lib.opattn_prefill_paged_plan_create.argtypes = [ctypes.POINTER(P), P, P, i32, i32, i32, i32, i32, i32,
                                                             i32]
            lib.opattn_plan_run_paged.restype = ctypes.c_int
            lib.opattn_plan_run_paged.argtypes = [P, P, P, P, P, i64, P, P, f32, P]
            lib.opattn_decode_schedule.restype = ctypes.c_int
            lib.opattn_decode_schedule.argtypes = [P, P, i32, i32, i32, i32, i32, P, i64, P,
                                                   ctypes.POINTER(i64), ctypes.POINTER(i32)]
            lib.opattn_decode_schedule_default.restype = ctypes.c_int
            lib.opattn_decode_schedule_default.argtypes = [P, P, i32, i32, i32, i32, i32, P, i64, P,
                                                           ctypes.POINTER(i64), ctypes.POINTER(i32)]
            _lib = lib
    return _lib


def status_string(status: int) -> str:
    return load().opattn_status_string(int(status)).decode()


def opattn_version() -> int:
    return int(load().opattn_version())


def _cu(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _np_ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dptr(t):
    """Device pointer of a torch tensor (or an int address, or None)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream_handle(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def opattn_prefill(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int,
                   scale: float, stream=None, *, check: bool = True) -> int:
    """C ``opattn_prefill``: q/k/v/o/lse are CUDA tensors (or raw device addresses),
    cu_seqlens_* host int32 arrays of n_seq + 1 offsets.  Raises OpattnError unless
    check=False, in which case the status code is returned."""
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    st = load().opattn_prefill(_dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), _np_ptr(cq), _np_ptr(ck),
                               int(n_seq), int(Hq), int(Hkv), int(d), float(scale), _stream_handle(stream))
    if check and st != OPATTN_OK:
        raise OpattnError(st, "opattn_prefill")
    return st


def opattn_prefill_noalloc(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int,
                           scale: float, stream=None, *, check: bool = True) -> int:
    """C ``opattn_prefill_noalloc``: same arguments as opattn_prefill, but the library
    allocates no device memory (its work list goes to a fixed ~1.7 MB device array
    shared by all calls; see include/opattn.h).  For callers that cannot let a
    library allocate, e.g. an engine that has reserved nearly all HBM for its own
    pool.  Calls that overlap on the GPU race on the shared array."""
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    st = load().opattn_prefill_noalloc(_dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), _np_ptr(cq),
                                       _np_ptr(ck), int(n_seq), int(Hq), int(Hkv), int(d), float(scale),
                                       _stream_handle(stream))
    if check and st != OPATTN_OK:
        raise OpattnError(st, "opattn_prefill_noalloc")
    return st


def opattn_prefill_checked(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq: int, Hq: int, Hkv: int,
                           d: int, scale: float, stream=None, flags: int = 0) -> int:
    """C ``opattn_prefill_checked`` (synchronous; returns the status code)."""
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    return int(load().opattn_prefill_checked(_dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), _np_ptr(cq),
                                             _np_ptr(ck), int(n_seq), int(Hq), int(Hkv), int(d), float(scale),
                                             _stream_handle(stream), int(flags)))


def _schedule(fn_name: str, width: int, cu_seqlens_q, cu_seqlens_k, Hq: int, Hkv: int, d: int, n_ctas: int):
    lib = load()
    fn = getattr(lib, fn_name)
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    n_seq = len(cq) - 1
    n_units, n_used = ctypes.c_int64(0), ctypes.c_int32(0)
    st = fn(_np_ptr(cq), _np_ptr(ck), n_seq, Hq, Hkv, d, n_ctas, None, 0, None, ctypes.byref(n_units),
            ctypes.byref(n_used))
    if st not in (OPATTN_OK, OPATTN_ERR_CAPACITY):
        raise OpattnError(st, fn_name)
    units = np.zeros((max(n_units.value, 1), width), dtype=np.int32)
    offs = np.zeros(max(n_used.value, 0) + 1, dtype=np.int32)
    st = fn(_np_ptr(cq), _np_ptr(ck), n_seq, Hq, Hkv, d, n_ctas, _np_ptr(units), units.shape[0], _np_ptr(offs),
            ctypes.byref(n_units), ctypes.byref(n_used))
    if st != OPATTN_OK:
        raise OpattnError(st, fn_name)
    return units[:n_units.value], offs


def opattn_schedule(cu_seqlens_q, cu_seqlens_k, Hq: int, Hkv: int, d: int, n_ctas: int):
    """C ``opattn_schedule`` (host only).  Returns (units [n, 13] int32, cta_offsets [n_ctas_used + 1])."""
    return _schedule("opattn_schedule", len(UNIT_FIELDS), cu_seqlens_q, cu_seqlens_k, Hq, Hkv, d, n_ctas)


def opattn_decode_schedule_default(cu_seqlens_q, cu_seqlens_k, Hq: int, Hkv: int, d: int, sms: int):
    """C ``opattn_decode_schedule_default`` (host only): the schedule of the default decode grid on a
    device with ``sms`` SMs.  Returns (units [n, 12] int32, cta_offsets)."""
    return _schedule("opattn_decode_schedule_default", len(DEC_UNIT_FIELDS), cu_seqlens_q, cu_seqlens_k, Hq, Hkv,
                     d, sms)


def opattn_decode_schedule(cu_seqlens_q, cu_seqlens_k, Hq: int, Hkv: int, d: int, n_ctas: int):
    """C ``opattn_decode_schedule`` (host only).  Returns (units [n, 12] int32, cta_offsets)."""
    return _schedule("opattn_decode_schedule", len(DEC_UNIT_FIELDS), cu_seqlens_q, cu_seqlens_k, Hq, Hkv, d,
                     n_ctas)


def opattn_decode(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int,
                  scale: float, stream=None, *, check: bool = True) -> int:
    """C ``opattn_decode``: the arguments and results of opattn_prefill, for batches
    with few query tokens per sequence (Lq * Hq / Hkv <= 32, d = 128)."""
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    st = load().opattn_decode(_dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), _np_ptr(cq), _np_ptr(ck),
                              int(n_seq), int(Hq), int(Hkv), int(d), float(scale), _stream_handle(stream))
    if check and st != OPATTN_OK:
        raise OpattnError(st, "opattn_decode")
    return st


def opattn_decode_checked(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int,
                          scale: float, stream=None, flags: int = 0) -> int:
    """C ``opattn_decode_checked`` (synchronous; returns the status code)."""
    cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
    return int(load().opattn_decode_checked(_dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), _np_ptr(cq),
                                            _np_ptr(ck), int(n_seq), int(Hq), int(Hkv), int(d), float(scale),
                                            _stream_handle(stream), int(flags)))


def opattn_prefill_paged(q, k_cache, v_cache, block_table, num_blocks: int, block_size: int, max_blocks: int, o,
                         lse, cu_seqlens_q, seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int, scale: float,
                         stream=None, *, check: bool = True) -> int:
    """C ``opattn_prefill_paged``: the prefill kernel over paged K/V caches."""
    cq, lk = _cu(cu_seqlens_q), _cu(seqlens_k)
    st = load().opattn_prefill_paged(_dptr(q), _dptr(k_cache), _dptr(v_cache), _dptr(block_table),
                                     int(num_blocks), int(block_size), int(max_blocks), _dptr(o), _dptr(lse),
                                     _np_ptr(cq), _np_ptr(lk), int(n_seq), int(Hq), int(Hkv), int(d), float(scale),
                                     _stream_handle(stream))
    if check and st != OPATTN_OK:
        raise OpattnError(st, "opattn_prefill_paged")
    return st


def opattn_decode_paged(q, k_cache, v_cache, block_table, num_blocks: int, block_size: int, max_blocks: int, o, lse,
                        cu_seqlens_q, seqlens_k, n_seq: int, Hq: int, Hkv: int, d: int, scale: float, stream=None,
                        *, check: bool = True) -> int:
    """C ``opattn_decode_paged``: decode over paged K/V caches [num_blocks, block_size, Hkv, d]
    with a device block table [n_seq, max_blocks] and host key counts ``seqlens_k``."""
    cq, lk = _cu(cu_seqlens_q), _cu(seqlens_k)
    st = load().opattn_decode_paged(_dptr(q), _dptr(k_cache), _dptr(v_cache), _dptr(block_table), int(num_blocks),
                                    int(block_size), int(max_blocks), _dptr(o), _dptr(lse), _np_ptr(cq),
                                    _np_ptr(lk), int(n_seq), int(Hq), int(Hkv), int(d), float(scale),
                                    _stream_handle(stream))
    if check and st != OPATTN_OK:
        raise OpattnError(st, "opattn_decode_paged")
    return st


class Plan:
    """C ``opattn_plan_*``: a work list built and uploaded once, run many times.

    ``decode=True`` builds the plan for the decode kernel; ``block_size > 0``
    builds a paged plan (``cu_seqlens_k`` is then the per-sequence key counts)
    that runs with ``run_paged``.  Run, info and destroy are shared.
    """

    def __init__(self, cu_seqlens_q, cu_seqlens_k, Hq: int, Hkv: int, d: int, max_ctas: int = 0,
                 decode: bool = False, block_size: int = 0, max_blocks: int = 0):
        lib = load()
        cq, ck = _cu(cu_seqlens_q), _cu(cu_seqlens_k)
        self._h = ctypes.c_void_p()
        self.decode = decode
        self.paged = block_size > 0
        if self.paged:
            # paged plans take per-sequence key counts in place of cu_seqlens_k
            name = "opattn_decode_paged_plan_create" if decode else "opattn_prefill_paged_plan_create"
            st = getattr(lib, name)(ctypes.byref(self._h), _np_ptr(cq), _np_ptr(ck), len(cq) - 1, Hq, Hkv, d,
                                    block_size, max_blocks, max_ctas)
        else:
            name = "opattn_decode_plan_create" if decode else "opattn_plan_create"
            create = lib.opattn_decode_plan_create if decode else lib.opattn_plan_create
            st = create(ctypes.byref(self._h), _np_ptr(cq), _np_ptr(ck), len(cq) - 1, Hq, Hkv, d, max_ctas)
        if st != OPATTN_OK:
            raise OpattnError(st, name)
        n_units, n_ctas = ctypes.c_int64(0), ctypes.c_int32(0)
        lib.opattn_plan_info(self._h, ctypes.byref(n_units), ctypes.byref(n_ctas))
        self.n_units, self.n_ctas = n_units.value, n_ctas.value

    def run(self, q, k, v, o, lse, scale: float, stream=None) -> None:
        st = load().opattn_plan_run(self._h, _dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse), float(scale),
                                    _stream_handle(stream))
        if st != OPATTN_OK:
            raise OpattnError(st, "opattn_plan_run")

    def run_checked(self, q, k, v, o, lse, scale: float, stream=None, flags: int = 0) -> int:
        """C ``opattn_plan_run_checked`` (synchronous; returns the status code)."""
        return int(load().opattn_plan_run_checked(self._h, _dptr(q), _dptr(k), _dptr(v), _dptr(o), _dptr(lse),
                                                  float(scale), _stream_handle(stream), int(flags)))

    def run_paged(self, q, k_cache, v_cache, block_table, num_blocks: int, o, lse, scale: float, stream=None) -> None:
        st = load().opattn_plan_run_paged(self._h, _dptr(q), _dptr(k_cache), _dptr(v_cache), _dptr(block_table),
                                          int(num_blocks), _dptr(o), _dptr(lse), float(scale), _stream_handle(stream))
        if st != OPATTN_OK:
            raise OpattnError(st, "opattn_plan_run_paged")

    def close(self) -> None:
        if self._h:
            st = load().opattn_plan_destroy(self._h)
            self._h = ctypes.c_void_p()
            if st != OPATTN_OK:
                raise OpattnError(st, "opattn_plan_destroy")

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            if self._h:
                load().opattn_plan_destroy(self._h)
        except Exception:
            pass


def prefill(q, k, v, cu_seqlens_q, cu_seqlens_k, scale: float | None = None, stream=None):
    """Allocate O and LSE with torch and run opattn_prefill on CUDA tensors q [Tq,Hq,d], k/v [Tk,Hkv,d]."""
    import torch
    Tq, Hq, d = q.shape
    Hkv = k.shape[1]
    o = torch.empty((Tq, Hq, d), dtype=torch.bfloat16, device=q.device)
    lse = torch.empty((Tq, Hq), dtype=torch.float32, device=q.device)
    n_seq = len(cu_seqlens_q) - 1
    opattn_prefill(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d,
                   scale if scale is not None else d ** -0.5, stream)
    return o, lse


def decode(q, k, v, cu_seqlens_q, cu_seqlens_k, scale: float | None = None, stream=None):
    """Allocate O and LSE with torch and run opattn_decode on CUDA tensors q [Tq,Hq,d], k/v [Tk,Hkv,d]."""
    import torch
    Tq, Hq, d = q.shape
    Hkv = k.shape[1]
    o = torch.empty((Tq, Hq, d), dtype=torch.bfloat16, device=q.device)
    lse = torch.empty((Tq, Hq), dtype=torch.float32, device=q.device)
    n_seq = len(cu_seqlens_q) - 1
    opattn_decode(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d,
                  scale if scale is not None else d ** -0.5, stream)
    return o, lse
