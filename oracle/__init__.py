"""fp64 CPU oracle for MoNe test-time learning — test infrastructure only.

Imported by tests, ``__graft_entry__.smoke()`` and the benchmark's CPU
baseline leg; never by the product path.  See ``mone_oracle`` for the paper
map, the readings it takes and which functions are pinned.
"""
from .mone_oracle import *  # noqa: F401,F403
from .mone_oracle import (PLAIN, PAPER, Hyper, Meta, State, init_state, ttl_segment, ttl_context,
                          generate_kv, segment_gradient, segment_loss, memory_forward, transform_inputs,
                          token_rates, momentum_decay, silu, silu_prime, sigmoid, softplus, f64, row_norms,
                          attention)
