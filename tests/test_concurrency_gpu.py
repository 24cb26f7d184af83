"""Determinism and thread safety of the library (GPU).

Both kernels follow a schedule fixed by the batch and merge split key ranges
in a fixed order, so repeated runs give bitwise-identical outputs.  Host
threads calling the one-shot entry points at once, each on its own stream
(sharing the pinned staging pool and the tensor-map encoder), get the same
bits as a lone call.
"""
import threading

import pytest
import torch

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_13499_gb300 import build as pbuild
    pbuild.build()
    pkg.load()


PREFILL = W.Workload("det_prefill", [300, 1000, 45], [300, 1500, 45], 32, 8, 128, 1.0, 21)
DECODE = W.Workload("det_decode", [1, 2, 1], [30000, 9000, 640], 16, 2, 128, 1.0, 22)
SPLIT = W.Workload("det_split", [200], [20000], 16, 4, 128, 1.0, 23)  # prefill units cut into pieces


def outputs(w):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
    return o, lse


@pytest.mark.parametrize("w,decode", [(PREFILL, False), (DECODE, True), (SPLIT, False)],
                         ids=["prefill", "decode", "prefill_split"])
def test_repeated_runs_are_bitwise_identical(w, decode):
    q, k, v = W.make_inputs(w, "cuda")
    runs = []
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=decode) as plan:
        if decode or w is SPLIT:
            assert plan.n_units > w.n_seq * w.Hkv * (1 if decode else 4)  # split key ranges, merged in-kernel
        for _ in range(3):
            o, lse = outputs(w)
            plan.run(q, k, v, o, lse, w.scale)
            torch.cuda.synchronize()
            runs.append((o.clone(), lse.clone()))
    for o, lse in runs[1:]:
        assert torch.equal(o.view(torch.int16), runs[0][0].view(torch.int16))
        assert torch.equal(lse.view(torch.int32), runs[0][1].view(torch.int32))


def test_concurrent_host_threads_match_a_lone_call():
    cases = (("prefill", PREFILL), ("decode", DECODE), ("split", SPLIT))
    inputs = {name: W.make_inputs(w, "cuda") for name, w in cases}
    calls = {"prefill": pkg.opattn_prefill, "decode": pkg.opattn_decode, "split": pkg.opattn_prefill}
    ref = {}
    for name, w in cases:
        o, lse = outputs(w)
        calls[name](*inputs[name], o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
        torch.cuda.synchronize()
        ref[name] = (o, lse)
    errors = []

    def worker(tid):
        try:
            stream = torch.cuda.Stream()
            with torch.cuda.stream(stream):
                for it in range(6):
                    name, w = cases[(tid + it) % 3]
                    o, lse = outputs(w)
                    calls[name](*inputs[name], o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale,
                                stream)
                    stream.synchronize()
                    if not (torch.equal(o.view(torch.int16), ref[name][0].view(torch.int16))
                            and torch.equal(lse.view(torch.int32), ref[name][1].view(torch.int32))):
                        errors.append(f"thread {tid} call {it} ({name}) differs")
        except Exception as e:  # noqa: BLE001 - reported below
            errors.append(f"thread {tid}: {e!r}")

    threads = [threading.Thread(target=worker, args=(t,)) for t in range(4)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not any(t.is_alive() for t in threads)
    assert not errors, errors


def test_calls_queued_far_ahead_of_the_gpu_are_correct():
    """48 one-shot calls queued behind a kernel that keeps the GPU busy: the host runs more calls
    ahead than the staging pool holds buffers (32), so later calls wait for the oldest work-list
    upload and reuse its buffer.  Every call's output must equal a lone call's."""
    w = PREFILL
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, l_ref = outputs(w)
    pkg.opattn_prefill(q, k, v, o_ref, l_ref, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    outs = [outputs(w) for _ in range(48)]
    torch.cuda.synchronize()
    torch.cuda._sleep(400_000_000)  # ~0.2 s of GPU time ahead of the calls
    for o, lse in outs:
        pkg.opattn_prefill(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    for i, (o, lse) in enumerate(outs):
        assert torch.equal(o.view(torch.int16), o_ref.view(torch.int16)), f"call {i}: O differs"
        assert torch.equal(lse.view(torch.int32), l_ref.view(torch.int32)), f"call {i}: LSE differs"
