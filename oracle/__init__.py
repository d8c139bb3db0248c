"""CPU oracle for the RhymeFlow asynchronous denoising step core.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports this package:
only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may use it.  It shares no code with the CUDA library and
imports nothing from it.  Inputs come from the seeded generators in
``workloads``, which hold none of the method's arithmetic.

Everything is plain, slow fp64 numpy (pure Python loops for the schedule).
"""
from .rf_oracle import (  # noqa: F401
    sigmas, schedule, active_set_alg2, compact, project, attention, euler,
    sampler, flops_attn, keyframe_select, project_kv_cache, attention_block_masked, to_f64,
)
