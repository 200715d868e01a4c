"""libmilesloss: the per-token RL loss over the vocabulary (forward and
backward) as hand-written CUDA for GB300 (sm_103a), behind a C ABI
(``include/milesloss.h``). This package holds the CUDA sources (``csrc/``),
the in-tree build (``build.py``), the thin ctypes binding (``milesloss.py``),
a tensor-level convenience layer (``api.py``) and the seeded synthetic
workload generator (``workloads.py``)."""

from .milesloss import (  # noqa: F401
    RL_BF16,
    RL_F32,
    MilesLossError,
    RlLossParams,
    load,
    make_params,
    parse_stats,
    rl_loss_bwd,
    rl_loss_check_device_error,
    rl_loss_fwd,
    rl_loss_fwd_bwd,
    rl_loss_fwd_bwd_rows,
    rl_loss_workspace_size,
    rl_set_sweep_events,
    status_string,
)
