"""Seeded synthetic workloads shaped like the paper's user / risk-event graphs.

The paper's data set (a proprietary payment-risk graph, Section 4.1) is not available, so every
input here is synthetic: a two-type heterogeneous graph (users, risk events; Section 2.2) with
typed relations and their inverses, power-law out- and in-degrees, N(0,1) node features, Xavier
weights and an overlap set of long-tail nodes shared with a neighbouring subgraph (Section 3.1).

This module holds none of the method's arithmetic (no aggregation, projection, normalisation or
loss).  Both the CUDA path (tests, bench, smoke) and the CPU oracle read their inputs from here,
so the two sides see identical numbers.
"""
from .graphs import (  # noqa: F401
    RELATIONS,
    TEMPORAL_WINDOW,
    WORKLOADS,
    GraphSpec,
    Workload,
    bf16_round,
    make_context,
    make_graph,
    make_head_params,
    make_hgt_params,
    make_labels,
    make_layer_params,
    make_ring_part,
    make_temporal_params,
    make_workload,
    ring_ids,
    spec,
)
