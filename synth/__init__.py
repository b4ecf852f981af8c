"""Seeded synthetic workloads for the ReSpec verify-and-draft step.

This package only draws inputs: token buffers with planted repeats, draft
trees, logits, bf16 Q/K/V, score tables and entropy histories.  It holds none
of the method's arithmetic (no entropy, no matching, no attention, no
acceptance), so both the CUDA path and the oracle can be fed from it without
sharing any of the computation they are compared on.
"""
from .workloads import (CONFIGS, Spec, Workload, bf16_bits, bf16_to_f32, build,  # noqa: F401
                        make, small_spec)
