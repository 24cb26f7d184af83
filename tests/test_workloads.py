"""The seeded generator: counter-based, device independent, and shaped as stated."""
import math

import numpy as np
import torch

from paper_2608_13499_gb300 import workloads as W


def test_tensor_draws_match_pure_python_splitmix64():
    for seed, stream in [(0, 0), (0, 2), (7, 4)]:
        z = W.draws(seed, stream, 1000, 16, "cpu")
        for i in range(16):
            assert (int(z[i]) & ((1 << 64) - 1)) == W.draw_py(seed, stream, 1000 + i)


def test_splitmix64_reference_values():
    # splitmix64 with state 0 advanced once: published first output 0xE220A8397B1DCDAF
    assert W.splitmix64_py(0x9E3779B97F4A7C15) == 0xE220A8397B1DCDAF


def test_normals_are_chunking_independent_and_roughly_standard():
    a = W.normal_bf16(0, 1, 100_000, "cpu", chunk=1 << 20)
    b = W.normal_bf16(0, 1, 100_000, "cpu", chunk=7777)
    assert torch.equal(a, b)
    x = a.float()
    assert abs(x.mean().item()) < 0.02 and abs(x.std().item() - 1) < 0.02
    assert float(a[5]) == float(torch.tensor(W.normal_py(0, 1, 5), dtype=torch.float32).to(torch.bfloat16))


def test_standard_workloads():
    t = W.tiny()
    assert t.total_q == 82 and t.q_lens == [1, 17, 64] and (t.Hq, t.Hkv, t.d) == (4, 2, 64)
    assert math.isclose(t.scale, 1 / 8)
    l8 = W.llama3_8b()
    assert l8.n_seq == 16 and all(16 <= x <= 8192 for x in l8.q_lens) and l8.input_scale == 0.5
    assert l8.q_lens == l8.k_lens
    l70 = W.llama3_70b()
    assert l70.total_q == 32768 and (l70.Hq, l70.Hkv, l70.d) == (64, 8, 128)
    b = W.bursty()
    assert b.q_lens[:2] == [32768, 32768] and b.q_lens[2:] == [256] * 30
    c = W.chunked()
    pre = np.array(c.k_lens) - 512
    assert c.q_lens == [512] * 64 and pre.min() >= 0 and pre.max() <= 16384


def test_make_inputs_shapes_and_input_scale():
    w = W.Workload("x", [3, 5], [4, 6], 4, 2, 64, input_scale=0.5, seed=3)
    q, k, v = W.make_inputs(w)
    assert q.shape == (8, 4, 64) and k.shape == (10, 2, 64) and v.shape == (10, 2, 64)
    assert q.dtype == torch.bfloat16
    full = W.normal_bf16(3, W.STREAM_Q, 8 * 4 * 64, "cpu", 1.0)
    assert torch.equal(q.flatten(), (full.float() * 0.5).to(torch.bfloat16))


def test_paged_layout_round_trip():
    """Every key row lands in its own page slot; gathering through the block table restores the packed rows."""
    import torch
    lens = [5, 0, 40, 17, 128, 129]
    for page in (8, 16, 64, 128):
        lay = W.paged_layout(lens, page, seed=3)
        n_pages = [(L + page - 1) // page for L in lens]
        assert lay.max_blocks == max(n_pages) and lay.block_table.shape == (len(lens), lay.max_blocks)
        used = np.concatenate([lay.block_table[s, :n] for s, n in enumerate(n_pages)])
        assert len(set(used.tolist())) == len(used) == sum(n_pages)       # no page shared
        assert used.min() >= 0 and used.max() < lay.num_blocks
        assert lay.num_blocks > sum(n_pages)                               # spare pages exist
        for s, n in enumerate(n_pages):
            assert np.all(lay.block_table[s, n:] == -1)
        x = torch.arange(sum(lens) * 2 * 3, dtype=torch.float32).view(sum(lens), 2, 3)
        cache = W.to_paged(x, lens, lay, fill=-5.0)
        assert cache.shape == (lay.num_blocks, page, 2, 3)
        rows = [cache[lay.block_table[s, j // page], j % page] for s, L in enumerate(lens) for j in range(L)]
        assert torch.equal(torch.stack(rows), x)
        assert int((cache == -5.0).all(dim=-1).all(dim=-1).sum()) == lay.num_blocks * page - sum(lens)
