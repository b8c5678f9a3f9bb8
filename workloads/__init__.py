"""Seeded synthetic inputs for batched speculative verification.

This module only draws inputs; it holds none of the verification, allocation
or commit arithmetic.  Both the CPU oracle's tests and the CUDA path's tests
and benchmark take their inputs from here, so the two sides always see the
same bytes.
"""
from .synth import CONFIGS, DraftInputs, Workload, make, make_draft, pack_rows, budget_candidates

__all__ = ["CONFIGS", "DraftInputs", "Workload", "make", "make_draft", "pack_rows", "budget_candidates"]
