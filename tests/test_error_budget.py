"""CPU checks of the decode error budget (tests/budget.py) that the GPU
parity tests assert element by element.

1. The oracle's weighted spreads of V (dev, absv) equal the same sums
   recomputed here from the oracle's weights with numpy, and their closed
   forms for one and two tokens.
2. Bound (1) of tests/budget.py holds for a simulation of the kernel's
   arithmetic: tokens split into chunks with their own running maxima (the
   kernel's stages, warps and split-K items), each weight 2^(x - m_chunk)
   rounded to bf16 and added to both the numerator and the normaliser, the
   chunks merged with factors 2^(m_c - M).  Any split gives the same bound,
   so the simulated outputs of two splits differ by at most twice the budget
   (the GPU split-invariance test asserts exactly that).
3. At the shapes the GPU tests use, the simulated error stays below 5e-3
   (max) and 5e-4 (mean), and the budget itself below the contract's 1e-2.
4. The masked prefill kernel's lazy maximum (weights kept with an old
   maximum up to a row sum of 2^16, or redone after a raise) keeps bound (1).
"""
import math

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from synthetic import bf16_bits, bf16_normal
from tests.budget import U_BF16, decode_budget


def widen(bits):
    return torch.from_numpy(bits.astype(np.int16).copy()).view(torch.bfloat16).double().numpy()


def qkv(seed, n, Hq, Hkv, d, kscale=1.0):
    q = bf16_bits(bf16_normal((Hq, d), seed))
    k = bf16_bits(bf16_normal((n, Hkv, d), seed + 1, scale=kscale))
    v = bf16_bits(bf16_normal((n, Hkv, d), seed + 2))
    return q, k, v


def simulate_kernel(q, k, v, scale, chunks):
    """The kernel's weight rounding, in float64 elsewhere.  `chunks` lists
    the token boundaries of the partials (each with its own maximum)."""
    Hq, d = q.shape
    n, Hkv, _ = k.shape
    G = Hq // Hkv
    qf, kf, vf = widen(q), widen(k), widen(v)
    out = np.zeros((Hq, d))
    for h in range(Hq):
        g = h // G
        x = (kf[:, g, :] @ qf[h]) * scale * math.log2(math.e)   # log2 domain
        parts = []
        for a, b in zip(chunks[:-1], chunks[1:]):
            m = x[a:b].max()
            p = np.exp2(x[a:b] - m)
            pr = torch.from_numpy(p).to(torch.bfloat16).double().numpy()
            parts.append((m, pr.sum(), pr @ vf[a:b, g, :]))
        M = max(m for m, _, _ in parts)
        num = sum(np.exp2(m - M) * o for m, _, o in parts)
        den = sum(np.exp2(m - M) * l for m, l, _ in parts)
        out[h] = num / den
    return out


@pytest.mark.parametrize("n,Hq,Hkv,d", [(1, 4, 2, 64), (2, 16, 1, 64), (37, 8, 2, 128),
                                        (300, 32, 8, 128)])
def test_spreads_match_numpy(n, Hq, Hkv, d):
    q, k, v = qkv(n * 7 + d, n, Hq, Hkv, d)
    scale = 1.0 / math.sqrt(d)
    out, w = oatt.decode(q, k, v, scale, want_weights=True)
    out2, dev, absv = oatt.decode_dev(q, k, v, scale)
    assert np.array_equal(out, out2)
    vf = widen(v)
    G = Hq // Hkv
    for h in range(Hq):
        g = h // G
        np.testing.assert_allclose(dev[h], w[h] @ np.abs(vf[:, g, :] - out[h]), rtol=1e-12,
                                   atol=1e-14)
        np.testing.assert_allclose(absv[h], w[h] @ np.abs(vf[:, g, :]), rtol=1e-12, atol=1e-14)


def test_spreads_closed_forms():
    # one token: o = v, so dev = 0 and absv = |v|
    q, k, v = qkv(3, 1, 4, 2, 64)
    out, dev, absv = oatt.decode_dev(q, k, v, 0.125)
    assert np.all(dev == 0.0)
    vf = widen(v)
    for h in range(4):
        assert np.array_equal(absv[h], np.abs(vf[0, h // 2]))
    # two tokens with weights (a, 1 - a): dev = 2 a (1 - a) |v1 - v0|
    q, k, v = qkv(5, 2, 1, 1, 64)
    out, w = oatt.decode(q, k, v, 0.3, want_weights=True)
    _, dev, _ = oatt.decode_dev(q, k, v, 0.3)
    vf = widen(v)
    a = w[0, 0]
    np.testing.assert_allclose(dev[0], 2 * a * (1 - a) * np.abs(vf[1, 0] - vf[0, 0]), rtol=1e-12,
                               atol=1e-15)


# (n, G, d) of the GPU parity tests: ragged lengths around the page sizes,
# the merge-path contexts and the split-invariance context
SHAPES = [(1, 4, 64), (2, 16, 64), (15, 1, 64), (16, 4, 128), (17, 8, 128), (63, 16, 64),
          (64, 3, 64), (65, 6, 128), (199, 5, 128), (700, 4, 128), (2000, 1, 64),
          (3000, 3, 128), (9043, 4, 128)]


@pytest.mark.parametrize("n,G,d", SHAPES)
def test_budget_bounds_simulated_rounding(n, G, d):
    Hkv = 2
    q, k, v = qkv(n + 13 * G + d, n, G * Hkv, Hkv, d)
    scale = 1.0 / math.sqrt(d)
    exact, dev, absv = oatt.decode_dev(q, k, v, scale)
    rng = np.random.default_rng(n * 31 + G)
    bound = U_BF16 / (1 - U_BF16) * dev + 1e-12
    budget = decode_budget(dev, absv, n)
    sims = []
    for trial in range(3):
        # the kernel's partials: 16-token warp slices, then a random split
        cuts = set(range(0, n, 16)) | {n}
        cuts |= set(int(c) for c in rng.integers(1, n, size=min(n - 1, 5 * trial))) if n > 1 else set()
        chunks = sorted(cuts)
        sim = simulate_kernel(q, k, v, scale, chunks)
        err = np.abs(sim - exact)
        assert np.all(err <= bound), float((err / np.maximum(bound, 1e-30)).max())
        assert err.max() < 5e-3 and err.mean() < 5e-4
        sims.append(sim)
    for s in sims[1:]:
        assert np.all(np.abs(s - sims[0]) <= 2 * budget)
    assert budget.max() < 1e-2


def simulate_prefill_row(x, vf, tile=128, force=None):
    """The masked prefill kernel's weights for one query row, in float64
    elsewhere: key tiles of `tile` keys; a tile's weights 2^(x - m) with the
    running maximum m are rounded to bf16 and accepted while their (rounded)
    sum stays at most 2^16; otherwise the tile's maximum raises m where it
    grew by more than 2^8, O and the normaliser are rescaled and the tile is
    redone.  `force` (a generator) sometimes takes the second path although
    the row's own sum was small, as a row does when another row of its warp
    needs it.  Returns (output, accepted tiles whose largest weight exceeded
    1, raises after the first tile)."""
    m, l = -math.inf, 0.0
    o = np.zeros(vf.shape[1])
    above_one = raises = 0
    for a in range(0, len(x), tile):
        xt = x[a:a + tile]
        if m != -math.inf:
            pr = torch.from_numpy(np.exp2(xt - m)).to(torch.bfloat16).double().numpy()
            if pr.sum() <= 2.0 ** 16 and not (force is not None and force.random() < 0.1):
                above_one += int(pr.max() > 1.0)
                l += pr.sum()
                o += pr @ vf[a:a + tile]
                continue
        mt = xt.max()
        if mt > m + 8.0:
            alpha = 0.0 if m == -math.inf else 2.0 ** (m - mt)
            raises += int(m != -math.inf)
            m = mt
            l *= alpha
            o *= alpha
        pr = torch.from_numpy(np.exp2(xt - m)).to(torch.bfloat16).double().numpy()
        l += pr.sum()
        o += pr @ vf[a:a + tile]
    return o / l, above_one, raises


@pytest.mark.parametrize("scale,regime", [(0.35, "kept"), (1.0, "both"), (4.0, "raised")])
def test_prefill_lazy_maximum_keeps_the_budget(scale, regime):
    # Queries of the last positions of a 1,100-token sequence with logits
    # whose maxima grow from key tile to key tile.  Weights kept with an old
    # maximum (up to a row sum of 2^16) and weights redone after a raise are
    # rounded alike, and the normaliser sums the rounded weights, so the
    # output stays a convex combination of V rows: bound (1) of
    # tests/budget.py holds whatever the maximum was.
    n, d = 1100, 128
    rng = np.random.default_rng(int(scale * 100))
    tot_above = tot_raises = 0
    for row in range(12):
        q, k, v = qkv(row * 17 + int(scale * 10), n, 1, 1, d)
        kf, vf = widen(k)[:, 0, :], widen(v)[:, 0, :]
        x = (kf @ widen(q)[0]) * scale * math.log2(math.e)
        exact, dev, _ = oatt.decode_dev(q, k, v, scale)
        sim, above, raises = simulate_prefill_row(x, vf, force=rng if row % 3 == 2 else None)
        tot_above += above
        tot_raises += raises
        bound = U_BF16 / (1 - U_BF16) * dev[0] + 1e-12
        assert np.all(np.abs(sim - exact[0]) <= bound)
    # the regimes the GPU test's scales are meant to reach
    if regime in ("kept", "both"):
        assert tot_above > 0
    if regime in ("both", "raised"):
        assert tot_raises > 0
    if regime == "kept":
        assert tot_raises == 0
