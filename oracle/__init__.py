"""fp64 CPU oracle for the fixed-cost drafting round (test infrastructure only).

This package is a plain, slow restatement of what the drafting round computes,
written from the paper's text in its own order and notation:

* views.py   -- the fixed-size context interface (Sec. 2.2): boundary state h,
                recent KV window, and the global summary (Eq. global-summary),
                maintained incrementally by the merge of App. A.2
                (Eq. summary-update).
* drafter.py -- the block-diffusion drafter forward (Sec. 2.3, App. A.1):
                boundary fusion, input slots, D Qwen3-style layers attending over
                [block; window; summary] (Eq. draft-context), frozen final norm
                and LM head (base logits z^(0)).
* sampler.py -- the low-rank Markov correction (Eq. markov) and sequential
                proposal sampling (Eq. proposal-factorization) with Gumbel-max
                over a Philox4x32-10 stream.
* verify.py  -- target-side verification of a drafted block (Eq. acceptance,
                Eq. residual, the bonus draw of Sec. 2.1).
* philox.py  -- Philox4x32-10 (Salmon et al., SC'11) from its published definition.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import
it; the CUDA library never does, and this package imports nothing from it.
Every function works in float64 on inputs upcast from the stored bf16/fp32
bytes, and never rounds an intermediate.
"""
from . import philox, views, drafter, sampler, verify  # noqa: F401
from .views import OracleState, state_init, view_update, full_summary, state_bytes_per_request  # noqa: F401
from .drafter import OracleWeights, draft_base_logits  # noqa: F401
from .sampler import sample_block, gumbel  # noqa: F401
from .verify import verify_block  # noqa: F401
