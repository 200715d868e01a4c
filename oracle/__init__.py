"""Float64 CPU oracle of the per-token RL loss over the vocabulary.

TEST INFRASTRUCTURE ONLY. This package is the slow, plainly written definition
that the CUDA library is checked against. Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it. The library (``paper_2609_08368_gb300``) never imports it, and it imports
nothing from the library: the two share no code.
"""

from .rl_loss_ref import (  # noqa: F401
    LossParams,
    widen_bf16,
    row_log_softmax,
    group_advantages,
    row_advantages,
    shape_advantages_opd,
    estimator_advantages,
    training_tokens_per_trajectory,
    opd_topk_estimate,
    sequence_objective,
    correction_ratio,
    token_objective,
    masked_token_mean,
    loss_stats,
    dlogits_rows,
    rl_loss,
    rl_loss_rows,
)
