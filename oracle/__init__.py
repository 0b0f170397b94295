"""CPU oracle of the ReTrace round (test infrastructure only).

Imported only by the tests, ``__graft_entry__.smoke()`` and the CPU-baseline
legs of ``bench.py``; the product path never uses it.
"""

from .retrace_oracle import (  # noqa: F401
    accepted_length,
    align,
    bf16_bits_to_f64,
    bf16_ulp,
    carried_rows,
    VARIANTS,
    commit,
    condition,
    conditioned_rows,
    correct,
    filtered_distribution,
    gate_fuse,
    LOWRANK_CORRECTION,
    LOWRANK_LATENT,
    lowrank_condition,
    retrace_round_lowrank,
    retrace_round,
    round_to_bf16,
    sigmoid,
    target_argmax,
    verify,
    verify_sampled,
)
