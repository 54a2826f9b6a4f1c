"""Float64 CPU oracle for the verify step of two-reasoner speculative decoding.

TEST INFRASTRUCTURE ONLY. This package is a plain, slow, obviously correct
restatement of what the GPU path computes, written from the paper
("Reasoning-aware Speculative Decoding for Efficient VLA Models in Autonomous
Driving", arxiv 2606.31160):

  rope.py       1D RoPE (Eq. rope-1d), 3D M-RoPE (Eqs. rope-3d, axis-assign,
                mrope-phase) and FlatRoPE (Eq. flatrope-proj), Sec. 3.3 / 4.2
  attention.py  causal GQA attention of the K+1 verify rows (Eq. verify, Sec. 3.2)
  accept.py     greedy longest-prefix acceptance + bonus (Eqs. accept, commit)
                and Leviathan/Chen rejection sampling (cited in Sec. 1 and 2)
  kv.py         KV-cache append and rollback to the committed length (Eq. commit)
  budget.py     per-segment attention mass and normalised entropy of the verify
                rows (Sec. 4.2, Table tab:attn-budget)

Only tests/, __graft_entry__.smoke() and bench.py (its cpu_baseline leg and
its --impl reference arm) may import it. The CUDA library and its Python
binding never import it and share no code with it: the two sides meet only
through the seeded input generators, which hold none of the method's
arithmetic.

Every function takes float64 numpy arrays (bf16 / fp32 inputs widened
exactly) and computes in float64. Parity status of each function is given in
its own docstring; all of them are pinned by tests/test_oracle_*.py.
"""

from .rope import (rope_frequencies, axis_assignment, mrope_apply, rope_1d,
                   rope_1d_matrix, flatrope_positions)
from .attention import verify_attention
from .accept import accept_greedy, accept_sample, argmax_lowest
from .kv import kv_append, kv_rollback
from .budget import attention_budget

__all__ = [
    "rope_frequencies", "axis_assignment", "mrope_apply", "rope_1d",
    "rope_1d_matrix", "flatrope_positions", "verify_attention",
    "accept_greedy", "accept_sample", "argmax_lowest", "kv_append",
    "kv_rollback", "attention_budget",
]
