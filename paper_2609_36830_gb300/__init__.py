"""PACE hot path on GB300: pool scoring, adaptive rejection and the fused
LM-head log-prob + clipped surrogate, as hand-written CUDA behind a C ABI.

``paper_2609_36830_gb300.pace`` is the Python binding of the C library;
``paper_2609_36830_gb300.workloads`` draws the seeded synthetic inputs.
Importing this package loads neither.
"""
__all__ = ["pace", "workloads"]
