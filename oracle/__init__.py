"""CPU oracle for the SideQuest KV-cache hot path.

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only tests/, __graft_entry__.smoke()
and bench.py's CPU-baseline / reference legs may import, call, link or run
anything in this package.  The CUDA library (paper_2602_22603_gb300) never
imports it, and it never imports the CUDA library: the two share no code,
header, table or constant; only the seeded input generators in `synthetic`
feed both.

Contents:
  cache_model  paged cache as an integer state machine (fork, append, evict,
               release; lowest-free-id allocation; copy-on-write rules).
  attention    decode attention in double precision over bf16 inputs
               (plain C, oracle/attention.c), with optional token mask;
               masked prefill attention (causal, span tokens removed:
               Algorithm 2's BuildMask) built on the same per-query routine.

Parity status: every function here is pinned by tests/test_oracle_pins.py
against closed forms, invariants, brute force and library routines; nothing
is "parity unpinned".
"""
from . import attention, cache_model  # noqa: F401
