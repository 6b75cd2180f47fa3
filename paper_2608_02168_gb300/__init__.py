"""GB300 (sm_103a) hot path of risk-aware overlapping-subgraph GNN training.

`hg` is the binding of the C-ABI library libhg.so (include/hg.h); `step.HotPath` drives one
training step of one subgraph through it.  The library must be built first
(`python -m paper_2608_02168_gb300.build`); nothing here falls back to another implementation.
"""
from . import hg  # noqa: F401
