"""Seeded synthetic inputs shared by the tests, the oracle checks and the bench.

This module only draws random numbers and lays out workload shapes. It holds
none of the method's arithmetic: no attention, no page-table rule, no
eviction rule.  Both the CUDA path and the CPU oracle consume what it makes.

Workload shapes stand in for the agentic contexts of the paper's evaluation
(Sec. 4.1, FRAMES / BrowseComp-Plus traces reaching past 100k tokens, Fig. 2):
only their length structure is imitated; no dataset item is reproduced.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np
import torch


# ---------------------------------------------------------------------------
# Workload shapes (one per benchmark configuration)
# ---------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Shape:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def bytes_per_token_layer(self) -> int:
        # K and V, bf16
        return 2 * self.num_kv_heads * self.head_dim * 2


TINY = Shape("tiny-1L-16q4kv-d64-P16", 1, 16, 4, 64, 16)
AGENT_8B = Shape("8b-32L-32q8kv-d128-P64", 32, 32, 8, 128, 64)
LARGE_70B = Shape("70b-80L-64q8kv-d128-P64", 80, 64, 8, 128, 64)


# ---------------------------------------------------------------------------
# Random tensors
# ---------------------------------------------------------------------------
def torch_gen(seed: int, device: str = "cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def sub_seed(seed: int, purpose: int) -> int:
    """Independent sub-stream for one purpose of one workload seed."""
    return int(seed) * 1000 + int(purpose)


def bf16_normal(shape: Sequence[int], seed: int, device: str = "cpu",
                scale: float = 1.0) -> torch.Tensor:
    """N(0,1) (times `scale`) drawn in fp32 from a seeded generator, rounded
    to bf16 (round-to-nearest-even, torch's default conversion)."""
    g = torch_gen(seed, device)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if scale != 1.0:
        x = x * scale
    return x.to(torch.bfloat16)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """The raw bf16 bit patterns of a CPU tensor as a uint16 numpy array."""
    assert t.dtype == torch.bfloat16
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


class Bank:
    """A large seeded N(0,1) bf16 buffer from which big workloads slice their
    K/V chunks at seeded offsets (so a 100+ GiB pool is filled without drawing
    100+ GiB of fresh normals; any row can be re-derived from its offset)."""

    def __init__(self, n_elems: int, seed: int, device: str = "cpu",
                 scale: float = 1.0):
        self.n_elems = int(n_elems)
        self.seed = int(seed)
        self.scale = float(scale)
        self.data = bf16_normal((self.n_elems,), seed, device=device, scale=scale)

    def offsets(self, count: int, chunk_elems: int, seed: int) -> np.ndarray:
        """`count` offsets, multiples of 8 elements (16 bytes), at which a
        chunk of `chunk_elems` fits inside the bank."""
        hi = (self.n_elems - chunk_elems) // 8
        assert hi > 0, "bank smaller than one chunk"
        rng = np.random.default_rng(seed)
        return rng.integers(0, hi, size=count, dtype=np.int64) * 8

    def view(self, offset: int, shape: Sequence[int]) -> torch.Tensor:
        n = int(np.prod(shape))
        return self.data[int(offset):int(offset) + n].view(*shape)


# ---------------------------------------------------------------------------
# Span layouts (stand-ins for cursor-identified tool responses)
# ---------------------------------------------------------------------------
def lognormal_lengths(rng: np.random.Generator, count: int, median: float,
                      sigma: float, total: Optional[int] = None,
                      cap: Optional[int] = None) -> np.ndarray:
    """`count` lognormal lengths (given median and sigma); if `total` is given
    they are rescaled to sum exactly to it by largest-remainder rounding, each
    kept >= 1."""
    x = rng.lognormal(mean=math.log(median), sigma=sigma, size=count)
    if cap is not None:
        x = np.minimum(x, cap)
    if total is None:
        return np.maximum(1, np.rint(x)).astype(np.int64)
    assert total >= count
    # reserve 1 per span, distribute the rest proportionally
    rest = total - count
    w = x / x.sum() * rest
    base = np.floor(w).astype(np.int64)
    rem = rest - int(base.sum())
    order = np.argsort(-(w - base), kind="stable")
    base[order[:rem]] += 1
    return base + 1


def place_spans(rng: np.random.Generator, lengths: Sequence[int], lo: int,
                hi: int) -> List[Tuple[int, int]]:
    """Place spans of the given lengths, in a random order, without overlap
    inside [lo, hi): the free tokens are split into len+1 gaps by a uniformly
    random composition (stars and bars).  Returns half-open (start, end)
    pairs sorted by start."""
    lengths = [int(x) for x in lengths]
    k = len(lengths)
    free = (hi - lo) - sum(lengths)
    assert free >= 0, "spans do not fit"
    # uniformly random composition of `free` into k+1 non-negative parts
    bars = np.sort(rng.choice(free + k, size=k, replace=False)) if k else np.array([], dtype=np.int64)
    gaps = []
    prev = -1
    for b in bars:
        gaps.append(int(b - prev - 1))
        prev = int(b)
    order = rng.permutation(k)
    spans = []
    pos = lo
    for i in range(k):
        pos += gaps[i]
        ln = lengths[int(order[i])]
        spans.append((pos, pos + ln))
        pos += ln
    return spans


def random_spans(seed: int, n_spans: int, total: int, lo: int, hi: int,
                 median: float, sigma: float = 0.75) -> List[Tuple[int, int]]:
    rng = np.random.default_rng(seed)
    lens = lognormal_lengths(rng, n_spans, median, sigma, total=total)
    return place_spans(rng, lens, lo, hi)


def shuffled(spans: Sequence[Tuple[int, int]], seed: int) -> List[Tuple[int, int]]:
    """The same spans in a seeded random order (the library accepts unsorted
    span lists)."""
    rng = np.random.default_rng(seed)
    idx = rng.permutation(len(spans))
    return [tuple(spans[int(i)]) for i in idx]


def request_spans(seed: int, r: int, n: int, P: int, frac=(0.20, 0.65), count=(10, 40),
                  median: float = 2000.0) -> List[Tuple[int, int]]:
    """Spans for one request of the batched-serving workload: a uniform
    fraction of the context in a uniform number of spans with lognormal
    lengths, inside [P, n), in shuffled order."""
    rng = np.random.default_rng(sub_seed(seed, 100 + r))
    f = rng.uniform(*frac)
    k = int(rng.integers(count[0], count[1] + 1))
    total = int(f * (n - P))
    return shuffled(random_spans(sub_seed(seed, 200 + r), k, total, P, n, median=median), r)
