"""C-ABI checks that need no GPU: the library loads, exports every declared
symbol, and rejects bad arguments on the host before any device work."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import build as pbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "opattn.h")


@pytest.fixture(scope="module")
def lib():
    pbuild.build()
    return pkg.load()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"OPATTN_API[^;(]*?\b(opattn_\w+)\s*\(", text)))


def test_header_declares_the_entry_points():
    syms = declared_symbols()
    for name in ["opattn_prefill", "opattn_prefill_checked", "opattn_prefill_noalloc", "opattn_plan_create",
                 "opattn_plan_run", "opattn_plan_run_checked", "opattn_plan_destroy", "opattn_plan_info", "opattn_schedule",
                 "opattn_decode", "opattn_decode_checked", "opattn_decode_plan_create", "opattn_decode_schedule",
                 "opattn_decode_schedule_default",
                 "opattn_decode_paged", "opattn_decode_paged_plan_create", "opattn_prefill_paged",
                 "opattn_prefill_paged_plan_create", "opattn_plan_run_paged", "opattn_version",
                 "opattn_status_string"]:
        assert name in syms, name


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
        assert isinstance(getattr(lib, name), ctypes._CFuncPtr)


def test_version_and_status_strings(lib):
    assert pkg.opattn_version() == 10100
    assert pkg.status_string(0) == "ok"
    for code in range(1, 7):
        assert pkg.status_string(code) not in ("ok", "unknown status")
    assert pkg.status_string(99) == "unknown status"


# Fake, never-dereferenced device addresses: validation must fail on the host
# before the library touches CUDA (this machine has no GPU).
A = 0x10000


def call(q=A, k=A, v=A, o=A, lse=A, cu_q=(0, 4), cu_k=(0, 4), n_seq=1, Hq=4, Hkv=2, d=64, scale=0.125):
    return pkg.opattn_prefill(q, k, v, o, lse, cu_q, cu_k, n_seq, Hq, Hkv, d, scale, stream=0, check=False)


def test_empty_batch_is_ok_without_device_work(lib):
    assert call(n_seq=0, cu_q=(0,), cu_k=(0,)) == pkg.OPATTN_OK
    assert call(cu_q=(0, 0), cu_k=(0, 5)) == pkg.OPATTN_OK  # total_q == 0
    assert call(q=None, o=None, lse=None, cu_q=(0, 0, 0), cu_k=(0, 0, 0), n_seq=2) == pkg.OPATTN_OK


@pytest.mark.parametrize("kwargs,status", [
    (dict(q=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(o=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(lse=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(k=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(Hq=6, Hkv=4), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(Hq=0), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(Hkv=-1), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(n_seq=-1), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(cu_q=(1, 4)), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(cu_q=(0, 4, 3), cu_k=(0, 4, 5), n_seq=2), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(cu_k=(0, 5, 2), cu_q=(0, 1, 2), n_seq=2), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(scale=0.0), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(scale=-0.125), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(scale=float("nan")), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(scale=float("inf")), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(d=96), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(d=256), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(Hq=256, Hkv=1), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(q=A + 8), pkg.OPATTN_ERR_MISALIGNED),
    (dict(k=A + 2), pkg.OPATTN_ERR_MISALIGNED),
    (dict(v=A + 4), pkg.OPATTN_ERR_MISALIGNED),
    (dict(o=A + 8), pkg.OPATTN_ERR_MISALIGNED),
    (dict(lse=A + 2), pkg.OPATTN_ERR_MISALIGNED),
])
def test_argument_errors(lib, kwargs, status):
    assert call(**kwargs) == status


def test_null_kv_allowed_when_no_keys(lib):
    # every row sees no key; k/v may be NULL.  The call needs the GPU after
    # validation, so only the pre-device checks are exercised: misaligned o
    # still reports MISALIGNED even with k = v = NULL.
    assert call(k=None, v=None, o=A + 8, cu_k=(0, 0)) == pkg.OPATTN_ERR_MISALIGNED


def test_checked_entry_rejects_unknown_flags(lib):
    st = pkg.opattn_prefill_checked(A, A, A, A, A, (0, 4), (0, 4), 1, 4, 2, 64, 0.125, stream=0, flags=0x80)
    assert st == pkg.OPATTN_ERR_INVALID_ARG


def test_plan_create_validates(lib):
    with pytest.raises(pkg.OpattnError) as e:
        pkg.Plan((0, 4), (0, 4), 4, 2, 80)
    assert e.value.status == pkg.OPATTN_ERR_UNSUPPORTED
    with pytest.raises(pkg.OpattnError) as e:
        pkg.Plan((0, 4, 2), (0, 4, 6), 4, 2, 64)
    assert e.value.status == pkg.OPATTN_ERR_INVALID_ARG


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    monkeypatch.setattr(pkg, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(pkg, "_lib", None)
    with pytest.raises(ImportError):
        pkg.load()
