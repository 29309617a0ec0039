"""CPU oracle of the X-Cache chunk step -- TEST INFRASTRUCTURE ONLY.

Plain, slow, obviously-correct numpy (fp64) restatement of what the GPU path
computes, written from the paper (X-Cache, arXiv 2604.20289, Sections 2.1-2.5
and Table 1).  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline leg may import it; the product package never does.  It shares no
code with the CUDA path: the only common module is ``xc_inputs`` (seeded
synthetic inputs, no method arithmetic).
"""
from .xcache_oracle import (  # noqa: F401
    GateParams, GateCell, OracleModel, OracleXCache, Decision,
    to_bf16, layer_norm, silu, gelu_tanh, timestep_embedding, rope_pair_table,
    apply_rope, token_positions, attention, grid_allocation, axis_indices,
    fingerprint_rows, cosine, max_token_deviation, gate_decide, rollout, SIGMAS,
    group_token_positions, linear_rows, group_fingerprint_rows, gate_metrics,
)
