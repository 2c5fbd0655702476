"""Seeded synthetic inputs for the candidate-scoring path (no scoring arithmetic)."""
from .configs import (CATEGORICAL, CONTINUOUS, INT_LOG, INT_UNIFORM, ORDER, WORKLOADS,
                      Clause, Param, Workload, seeds)
from .generate import (CLAUSE_DTYPE, NODE_DTYPE, NODE_LEAF, PARAM_DTYPE, Instance, warp_params,
                       clause_array, draw_configs, make_instance, space_array, stored_values)
from .rng import Stream, stream_seed
