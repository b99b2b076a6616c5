"""Float64 CPU oracle for Jacap's eviction pass (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this package. The CUDA library never uses it.
"""

from .jacap_oracle import (  # noqa: F401
    JacapParams,
    window_stats,
    window_covariance,
    pool_attention,
    sensitivity,
    response_variance,
    response_variance_full,
    head_weight,
    unit_weights,
    capacity_matrix,
    jacap_scores,
    select_topb,
    greedy_logdet_select,
    compact,
    oracle_unit,
    oracle_pass,
    unit_views,
)
from .decode_oracle import decode_run  # noqa: F401,E402
