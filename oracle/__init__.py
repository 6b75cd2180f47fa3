"""CPU oracle of the hot path (test infrastructure only; never imported by the product path)."""
from .hg_oracle import *  # noqa: F401,F403
from .hg_oracle import (  # noqa: F401
    align_backward, align_forward, build_csr, layer_backward, layer_backward_rows, layer_forward,
    layer_forward_rows, mean_aggregate, overlap_intersect, standardise, step, valid_edges,
)
from . import overlap_build  # noqa: F401  (overlapping-subgraph construction, Eq. 4-5)
from . import head  # noqa: F401  (MeanAgg, MLP head, masked BCE and joint objective, Eq. 18-20)
from . import temporal  # noqa: F401  (context attention over the last w states and the GRU cell, Eq. 12-13)
from . import hgt  # noqa: F401  (attention variant of the layer, Eq. 6-11)
