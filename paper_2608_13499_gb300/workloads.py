"""Seeded synthetic workloads for the prefill-attention operator.

This module holds no attention arithmetic: it only draws random numbers and
builds sequence-length tables.  The CUDA path and the fp64 oracle are both fed
from it, so both sides always see the same input bits.

Random numbers are counter based, so they do not depend on device, chunking
or thread count:

* ``splitmix64`` (Steele, Lea, Flood 2014) of ``base(seed, stream) + (i+1) *
  0x9E3779B97F4A7C15`` gives the 64-bit draw for element ``i``;
* the high and low 32-bit halves become two uniforms in (0, 1);
* Box-Muller (cosine branch) turns them into one N(0, 1) value in float64;
* the value is multiplied by the workload's input scale, rounded to float32
  and then to bfloat16 (round-to-nearest-even at each step).

Streams: q = 0, k = 1, v = 2, prompt lengths = 3, chunk prefixes = 4.

The workloads stand in for the production traces the paper replays (Azure and
Mooncake traces); their shapes follow the paper's prompt-length range
(128 to 64K tokens, §2.1) and the head shapes of Llama-3 8B and 70B.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

_MASK64 = (1 << 64) - 1
_GOLDEN = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB

STREAM_Q, STREAM_K, STREAM_V, STREAM_LEN, STREAM_PREFIX = 0, 1, 2, 3, 4


def _signed(x: int) -> int:
    x &= _MASK64
    return x - (1 << 64) if x >= (1 << 63) else x


def splitmix64_py(x: int) -> int:
    """splitmix64 finaliser on a Python int, modulo 2**64 (reference for the tensor form)."""
    z = x & _MASK64
    z = ((z ^ (z >> 30)) * _M1) & _MASK64
    z = ((z ^ (z >> 27)) * _M2) & _MASK64
    return z ^ (z >> 31)


def stream_base(seed: int, stream: int) -> int:
    return splitmix64_py((seed << 16) + stream)


def draw_py(seed: int, stream: int, i: int) -> int:
    """64-bit draw number i of (seed, stream), pure Python."""
    return splitmix64_py(stream_base(seed, stream) + (i + 1) * _GOLDEN)


def _srl(x: torch.Tensor, s: int) -> torch.Tensor:
    """Logical right shift of int64 bit patterns."""
    return (x >> s) & ((1 << (64 - s)) - 1)


def draws(seed: int, stream: int, start: int, n: int, device) -> torch.Tensor:
    """64-bit draws start..start+n-1 as int64 bit patterns (wrapping arithmetic)."""
    idx = torch.arange(start + 1, start + n + 1, dtype=torch.int64, device=device)
    z = idx * _signed(_GOLDEN) + _signed(stream_base(seed, stream))
    z = (z ^ _srl(z, 30)) * _signed(_M1)
    z = (z ^ _srl(z, 27)) * _signed(_M2)
    return z ^ _srl(z, 31)


def _normal_from_draws(z: torch.Tensor) -> torch.Tensor:
    hi = _srl(z, 32).to(torch.float64)
    lo = (z & 0xFFFFFFFF).to(torch.float64)
    u1 = (hi + 0.5) * (1.0 / 4294967296.0)
    u2 = (lo + 0.5) * (1.0 / 4294967296.0)
    return torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2)


def normal_bf16(seed: int, stream: int, n: int, device, scale: float = 1.0,
                chunk: int = 1 << 24) -> torch.Tensor:
    """n i.i.d. N(0, scale^2) values as bfloat16 (float64 -> float32 -> bfloat16)."""
    out = torch.empty(n, dtype=torch.bfloat16, device=device)
    for s0 in range(0, n, chunk):
        m = min(chunk, n - s0)
        x = _normal_from_draws(draws(seed, stream, s0, m, device))
        if scale != 1.0:
            x = x * scale
        out[s0:s0 + m] = x.to(torch.float32).to(torch.bfloat16)
    return out


def normal_py(seed: int, stream: int, i: int) -> float:
    z = draw_py(seed, stream, i)
    u1 = ((z >> 32) + 0.5) / 4294967296.0
    u2 = ((z & 0xFFFFFFFF) + 0.5) / 4294967296.0
    return math.sqrt(-2.0 * math.log(u1)) * math.cos(2.0 * math.pi * u2)


def uniform_py(seed: int, stream: int, i: int) -> float:
    return ((draw_py(seed, stream, i) >> 32) + 0.5) / 4294967296.0


@dataclass
class Workload:
    """One ragged batch: per-sequence query/key lengths plus head geometry."""
    name: str
    q_lens: list
    k_lens: list
    Hq: int
    Hkv: int
    d: int
    input_scale: float = 1.0
    seed: int = 0
    scale: float = field(default=0.0)
    page_size: int = 0  # > 0: the decode workload keeps K/V in a paged cache of this page size

    def __post_init__(self):
        if self.scale == 0.0:
            self.scale = 1.0 / math.sqrt(self.d)
        if len(self.q_lens) != len(self.k_lens):
            raise ValueError("q_lens and k_lens differ in length")

    @property
    def n_seq(self) -> int:
        return len(self.q_lens)

    @property
    def cu_q(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.q_lens)]).astype(np.int32)

    @property
    def cu_k(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.k_lens)]).astype(np.int32)

    @property
    def total_q(self) -> int:
        return int(sum(self.q_lens))

    @property
    def total_k(self) -> int:
        return int(sum(self.k_lens))

    def describe(self) -> dict:
        return {"workload": self.name, "n_seq": self.n_seq, "Hq": self.Hq, "Hkv": self.Hkv,
                "head_dim": self.d, "total_q": self.total_q, "total_k": self.total_k,
                "input_scale": self.input_scale, "seed": self.seed}


def make_inputs(w: Workload, device="cpu"):
    """(q, k, v) bf16 tensors [total, heads, d] on `device` for workload w."""
    q = normal_bf16(w.seed, STREAM_Q, w.total_q * w.Hq * w.d, device, w.input_scale)
    k = normal_bf16(w.seed, STREAM_K, w.total_k * w.Hkv * w.d, device, w.input_scale)
    v = normal_bf16(w.seed, STREAM_V, w.total_k * w.Hkv * w.d, device, w.input_scale)
    return (q.view(w.total_q, w.Hq, w.d), k.view(w.total_k, w.Hkv, w.d),
            v.view(w.total_k, w.Hkv, w.d))


# --------------------------------------------------------------------------
# The five standard workloads
# --------------------------------------------------------------------------

def tiny(seed: int = 0) -> Workload:
    """3 sequences {1, 17, 64}, Hq 4, Hkv 2, d 64, N(0,1): 82 query tokens."""
    lens = [1, 17, 64]
    return Workload("tiny_ragged_3seq_d64", lens, list(lens), 4, 2, 64, 1.0, seed)


def lognormal_lengths(seed: int, n: int, median: float = 1024.0, sigma: float = 0.8,
                      lo: int = 16, hi: int = 8192) -> list:
    """clamp(floor(median * exp(sigma * z) + 0.5), lo, hi) with z from stream 3."""
    out = []
    for i in range(n):
        z = normal_py(seed, STREAM_LEN, i)
        out.append(int(min(hi, max(lo, math.floor(median * math.exp(sigma * z) + 0.5)))))
    return out


def llama3_8b(seed: int = 0) -> Workload:
    """16 prompts, lognormal(median 1024, sigma 0.8) in [16, 8192]; Hq 32, Hkv 8, d 128; inputs x0.5."""
    lens = lognormal_lengths(seed, 16)
    return Workload("llama3_8b_ragged_16seq", lens, list(lens), 32, 8, 128, 0.5, seed)


def llama3_70b(seed: int = 0) -> Workload:
    """8 prompts of 4096 tokens; Hq 64, Hkv 8, d 128."""
    lens = [4096] * 8
    return Workload("llama3_70b_8x4096", lens, list(lens), 64, 8, 128, 1.0, seed)


def bursty(seed: int = 0) -> Workload:
    """2 prompts of 32768 tokens plus 30 of 256; Hq 32, Hkv 8, d 128."""
    lens = [32768] * 2 + [256] * 30
    return Workload("bursty_2x32k_30x256", lens, list(lens), 32, 8, 128, 1.0, seed)


def chunk_prefixes(seed: int, n: int, hi: int = 16384) -> list:
    """Uniform integers in [0, hi] (inclusive) from stream 4."""
    return [int(math.floor(uniform_py(seed, STREAM_PREFIX, i) * (hi + 1))) for i in range(n)]


def chunked(seed: int = 0) -> Workload:
    """64 chunks of 512 queries attending to prefix + 512 keys, prefix ~ U[0, 16384]."""
    pre = chunk_prefixes(seed, 64)
    return Workload("chunked_64x512_prefix16k", [512] * 64, [512 + p for p in pre],
                    32, 8, 128, 1.0, seed)


def decode_llama3_70b(seed: int = 0) -> Workload:
    """64 requests decoding one token each over 8192 cached keys; Hq 64, Hkv 8, d 128."""
    return Workload("decode_llama3_70b_64x8192", [1] * 64, [8192] * 64, 64, 8, 128, 1.0, seed)


def decode_llama3_8b(seed: int = 0) -> Workload:
    """128 requests decoding one token each over lognormal(median 4096, sigma 0.8) in [16, 32768]
    cached keys; Hq 32, Hkv 8, d 128."""
    lens = lognormal_lengths(seed, 128, median=4096.0, sigma=0.8, lo=16, hi=32768)
    return Workload("decode_llama3_8b_ragged_128seq", [1] * 128, lens, 32, 8, 128, 1.0, seed)


def decode_spec4_llama3_70b(seed: int = 0) -> Workload:
    """32 requests verifying 4 speculative tokens each over 16384 cached keys; Hq 64, Hkv 8, d 128."""
    return Workload("decode_spec4_llama3_70b_32x16384", [4] * 32, [16384] * 32, 64, 8, 128, 1.0, seed)


def decode_llama3_70b_paged16(seed: int = 0) -> Workload:
    """decode_llama3_70b with its K/V in a paged cache of 16-key pages in shuffled order."""
    w = Workload("decode_llama3_70b_paged16_64x8192", [1] * 64, [8192] * 64, 64, 8, 128, 1.0, seed)
    w.page_size = 16
    return w


DECODE = {"decode_llama3_70b": decode_llama3_70b, "decode_llama3_8b": decode_llama3_8b,
          "decode_spec4_llama3_70b": decode_spec4_llama3_70b, "decode_llama3_70b_paged16": decode_llama3_70b_paged16}


# --------------------------------------------------------------------------
# Paged K/V caches
# --------------------------------------------------------------------------

@dataclass
class PagedLayout:
    """Where each sequence's keys live in a paged cache [num_blocks, page_size, heads, d]."""
    page_size: int
    num_blocks: int
    block_table: np.ndarray  # int32 [n_seq, max_blocks]; -1 where a sequence has no page
    max_blocks: int


def paged_layout(k_lens, page_size: int, seed: int = 0, spare: float = 0.25) -> PagedLayout:
    """Give every sequence ceil(Lk / page_size) pages drawn in a seeded random order from a pool
    with `spare` unused pages, so that consecutive pages of a sequence are scattered."""
    n_pages = [(int(L) + page_size - 1) // page_size for L in k_lens]
    total = sum(n_pages)
    num_blocks = max(1, total + int(spare * total) + 1)
    perm = np.random.default_rng(seed).permutation(num_blocks).astype(np.int32)
    max_blocks = max([1] + n_pages)
    table = np.full((len(k_lens), max_blocks), -1, dtype=np.int32)
    off = 0
    for s, n in enumerate(n_pages):
        table[s, :n] = perm[off:off + n]
        off += n
    return PagedLayout(page_size, num_blocks, table, max_blocks)


def to_paged(x: torch.Tensor, k_lens, layout: PagedLayout, fill: float = 7.0) -> torch.Tensor:
    """Scatter packed rows x [total_k, heads, d] into a paged cache; every other row holds `fill`."""
    heads, d = x.shape[1], x.shape[2]
    cache = torch.full((layout.num_blocks, layout.page_size, heads, d), fill, dtype=x.dtype, device=x.device)
    flat = cache.view(layout.num_blocks * layout.page_size, heads, d)
    rows = []
    for s, L in enumerate(k_lens):
        j = np.arange(int(L), dtype=np.int64)
        rows.append(layout.block_table[s, j // layout.page_size].astype(np.int64) * layout.page_size
                    + j % layout.page_size)
    idx = torch.from_numpy(np.concatenate(rows) if rows else np.zeros(0, dtype=np.int64)).to(x.device)
    flat[idx] = x
    return cache

STANDARD = {"tiny": tiny, "llama3_8b": llama3_8b, "llama3_70b": llama3_70b,
            "bursty": bursty, "chunked": chunked}


# --------------------------------------------------------------------------
# Chunked prefill of few requests over long cached prefixes (split-KV)
# --------------------------------------------------------------------------

def chunk_long_prefix(seed: int = 0) -> Workload:
    """One request's 512-token prompt chunk attending to a 16384-token cached prefix (chunked
    prefill, the step a long prompt takes once its earlier chunks are in the cache); Llama-3-8B
    heads (Hq 32, Hkv 8, d 128).  Its 64 work units are fewer than the SMs."""
    return Workload("chunk_1x512_prefix16k", [512], [512 + 16384], 32, 8, 128, 1.0, seed)


def chunks_long_prefix(seed: int = 0) -> Workload:
    """Four requests' 512-token chunks over prefixes drawn uniformly from [8192, 16384]
    (stream 4); Llama-3-8B heads."""
    pre = [8192 + p for p in chunk_prefixes(seed, 4, hi=8192)]
    return Workload("chunks_4x512_prefix8k_16k", [512] * 4, [512 + p for p in pre], 32, 8, 128, 1.0, seed)


LONG_PREFIX = {"chunk_long_prefix": chunk_long_prefix, "chunks_long_prefix": chunks_long_prefix}
