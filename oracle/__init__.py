"""Reference oracle for the TwinKV audit and repair pass (arXiv 2608.27128).

TEST INFRASTRUCTURE ONLY: a plain fp64 CPU restatement of the paper's definitions
(Sec. 3.2 Eq. 1 and the twin relation, Eq. 2-3 and the standalone policy, Sec. 3.4
Eq. 4 and the orphan/donor repair rule).  Only the test suite, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import it.  The CUDA library and its
Python binding never import it.
"""
from .oracle import (  # noqa: F401
    audit,
    build,
    count,
    policy,
    policy_select,
    repair,
    repair_dedup,
    repair_f32,
    round_bf16,
    sim,
)
