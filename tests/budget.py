"""Error budget of the decode kernel's fp32 outputs against the exact
(double precision) oracle, derived from the kernel's arithmetic.

The kernel forms every softmax weight in fp32 relative to a running maximum,
rounds it to bf16 for the tensor-core PV product, and adds the SAME rounded
weights into the normaliser.  With exact weights w_t (sum 1), exact output
o = sum_t w_t v_t and rounded weights p_t (1 + d_t), |d_t| <= u, the kernel's
output is the convex combination sum_t w_t (1 + d_t) v_t / (1 + dbar) with
dbar = sum_t w_t d_t, so

    out - o = sum_t w_t d_t (v_t - o) / (1 + dbar)
    |out - o| <= u / (1 - u) * sum_t w_t |v_t - o|                    (1)

for every output element.  Rescaling by 2^(m_old - m_new) and the split-K
merge multiply numerator and denominator by the same factors, so (1) holds
for any split of the tokens.  u = 2^-8 is the unit roundoff of bf16: it
keeps 8 significant bits, and rounding to nearest errs by at most half a
unit in the last place, 2^-8 of the leading bit.  u is raised by 2^-12 for
the fp32 logits (a 128-term fp32 dot product and the scale perturb a weight
by far less than 2^-12 relatively) and the hardware exponential.  The
remaining fp32 error is the accumulation of O and of the normaliser: at most
one fp32 rounding (counted as 2^-22, two units, to cover truncating
tensor-core accumulation) per 64-token stage an item holds, plus a few for
the merge, each relative to sum_t w_t |v_t|.

The oracle supplies sum_t w_t |v_t - o| (dev) and sum_t w_t |v_t| (absv).
"""
from __future__ import annotations

import math

import numpy as np

U_BF16 = 2.0 ** -8
U_WEIGHT = U_BF16 + 2.0 ** -12   # bf16 rounding + fp32 logit / exp2 error
U_ACC = 2.0 ** -22               # per fp32 accumulation step (2 ulps)
STAGE_TOKENS = 64


def decode_budget(dev: np.ndarray, absv: np.ndarray, n: int) -> np.ndarray:
    """Per-element bound on |kernel fp32 output - exact output| for a
    sequence of n tokens (dev, absv from oracle.attention.decode_dev)."""
    steps = math.ceil(n / STAGE_TOKENS) + 32
    return U_WEIGHT / (1.0 - U_WEIGHT) * dev + steps * U_ACC * absv + 1e-6
