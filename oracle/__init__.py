"""fp64 CPU oracle of the KVpop decode hot path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.  The
CUDA library never imports, links or calls anything here, and nothing here
imports the CUDA library.
"""
from .kvpop_oracle import (  # noqa: F401
    HeadCache,
    OracleParams,
    gelu_erf,
    scorer_mlp,
    round_score,
    static_priority,
    prefill_head,
    prefill_head_streaming,
    attend_head,
)
