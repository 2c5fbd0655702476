"""The five synthetic candidate-scoring workloads.

Each workload stands in for one round of SCOOT's suggestion step (Algorithm 1):
a search space of inference-engine parameters (Table 1 and the parameter
discussion of Section 2 give the vLLM parameters and types), the known
constraints of the engine (the appendix on known constraints), a set of
observed configurations with synthetic objective values, a random forest
trained on a synthetic crash label, and a large pool of candidate
configurations to score.

Parameter kinds (the mixed space of Section 3): INT_UNIFORM, INT_LOG,
CATEGORICAL (booleans are categoricals of two), CONTINUOUS.  Candidates are
stored structure-of-arrays, one 32-bit word per parameter: integers and
category indices as int32, continuous values as float32 bit patterns.

A clause is "all guards hold => sum_t coef_t * x[param_t] >= rhs" over the
integer-valued parameters (Eq. 2).
"""
from __future__ import annotations

from dataclasses import dataclass, field

INT_UNIFORM, INT_LOG, CATEGORICAL, CONTINUOUS = 0, 1, 2, 3


@dataclass(frozen=True)
class Param:
    name: str
    kind: int
    lo: float = 0.0
    hi: float = 0.0
    n_choices: int = 0
    default: float = 0.0  # stored value of the engine's default configuration


@dataclass(frozen=True)
class Clause:
    guards: tuple  # ((param, value), ...) at most 2
    terms: tuple   # ((param, coef), ...) at most 4
    rhs: int


@dataclass(frozen=True)
class Workload:
    name: str
    params: tuple
    clauses: tuple
    n_obs: int
    n_cand: int
    n_obj: int
    acq: str             # "ei" or "ehvi"
    n_trees: int
    max_depth: int
    n_mc: int            # S, Monte-Carlo samples for EHVI (0 for EI)
    q: int
    noise_sd: float      # observation noise of the synthetic surfaces
    noise_rho: float     # correlation of the noise between objectives
    signs: tuple         # +1 maximise the surface, -1 the surface is a latency
    budget: tuple        # ((param, weight), ...) of the synthetic memory budget;
                         # also the trade-off axis shared by the objectives
    tradeoff: tuple = (1.0, -1.0)   # weight of the trade-off axis in each objective (M > 1)
    conflict_scale: float = 0.5     # weight of the per-objective part when M > 1
    infeasible_frac: float = 0.25   # share of observations labelled as crashes
    label_flip: float = 0.10        # crash-label noise (forces deep trees)
    fantasy: bool = False
    delta_num: int = 10   # Delta = delta_num / delta_den = 0.5 (Algorithm 1 start)
    delta_den: int = 20
    leaf_scale: int = 255
    notes: str = field(default="", compare=False)

    @property
    def d(self) -> int:
        return len(self.params)


def _vllm10(mnbt_lo: float, mnbt_hi: float, max_len: int):
    """Ten vLLM parameters: Table 1 plus gpu-memory-utilization."""
    params = (
        Param("tensor_parallel", INT_UNIFORM, 1, 4, default=1),
        Param("max_num_seqs", INT_LOG, 64, 8192, default=256),
        Param("max_num_batched_tokens", INT_LOG, mnbt_lo, mnbt_hi, default=4096),
        Param("block_size", CATEGORICAL, n_choices=3, default=1),          # {8,16,32}
        Param("scheduler_delay_factor", CONTINUOUS, 0.0, 2.0, default=0.0),
        Param("enable_chunked_prefill", CATEGORICAL, n_choices=2, default=0),
        Param("enable_prefix_caching", CATEGORICAL, n_choices=2, default=0),
        Param("disable_custom_all_reduce", CATEGORICAL, n_choices=2, default=0),
        Param("use_v2_block_manager", CATEGORICAL, n_choices=2, default=0),
        Param("gpu_memory_utilization", CONTINUOUS, 0.5, 0.95, default=0.9),
    )
    # Known constraints of vLLM (appendix): mnbt >= mns; chunked prefill and
    # prefix caching not both on; without chunked prefill mnbt >= max model len.
    clauses = (
        Clause((), ((2, 1), (1, -1)), 0),
        Clause(((5, 1),), ((6, -1),), 0),
        Clause(((5, 0),), ((2, 1),), max_len),
    )
    return params, clauses


TINY = Workload(
    name="tiny",
    params=(
        Param("max_num_seqs", INT_LOG, 1, 1024, default=32),
        Param("max_num_batched_tokens_div", INT_LOG, 1, 1024, default=16),
        Param("block_size", CATEGORICAL, n_choices=3, default=1),
        Param("gpu_memory_utilization", CONTINUOUS, 0.5, 0.95, default=0.9),
    ),
    # Reading: the tiny workload names no constraint; x0 >= x1 is the Eq. 2
    # form with one term pair.
    clauses=(Clause((), ((0, 1), (1, -1)), 0),),
    n_obs=16, n_cand=4096, n_obj=2, acq="ehvi", n_trees=16, max_depth=6,
    n_mc=32, q=1, noise_sd=0.01, noise_rho=0.0, signs=(-1, -1),
    budget=((0, 1.0), (1, 1.0)),
)

_P8 = (
    Param("tensor_parallel", INT_LOG, 1, 8, default=1),
    Param("max_num_seqs", INT_LOG, 64, 8192, default=256),
    Param("max_num_batched_tokens", INT_LOG, 64, 8192, default=2048),
    Param("swap_space", INT_LOG, 1, 64, default=4),
    Param("max_seq_len_to_capture", INT_LOG, 256, 8192, default=8192),
    Param("block_size", CATEGORICAL, n_choices=3, default=1),
    Param("enable_chunked_prefill", CATEGORICAL, n_choices=2, default=0),
    Param("scheduler_delay_factor", CONTINUOUS, 0.0, 2.0, default=0.0),
)

D8 = Workload(
    name="d8-ehvi2",
    params=_P8,
    clauses=(
        Clause((), ((2, 1), (1, -1)), 0),          # mnbt >= mns
        Clause(((6, 0),), ((2, 1),), 2048),        # no chunked prefill => mnbt >= 2048
    ),
    n_obs=64, n_cand=1 << 18, n_obj=2, acq="ehvi", n_trees=100, max_depth=10,
    n_mc=64, q=4, noise_sd=0.01, noise_rho=0.0, signs=(-1, -1),
    budget=((1, 1.0), (2, 0.5), (0, -0.5)),
)

# The token-budget range and the model length are set so that about 40% of a
# uniform pool fails the known constraints (checked by the tests).
_P10, _C10 = _vllm10(mnbt_lo=1024, mnbt_hi=65536, max_len=2560)

D10_EI = Workload(
    name="d10-ei",
    params=_P10, clauses=_C10,
    n_obs=128, n_cand=1 << 20, n_obj=1, acq="ei", n_trees=100, max_depth=12,
    n_mc=0, q=1, noise_sd=0.02, noise_rho=0.0, signs=(-1,),
    budget=((1, 1.0), (2, 0.5), (9, 1.0), (0, -0.5)),
)

D10_EHVI3 = Workload(
    name="d10-ehvi3",
    params=_P10, clauses=_C10,
    n_obs=200, n_cand=1 << 20, n_obj=3, acq="ehvi", n_trees=128, max_depth=12,
    n_mc=128, q=8, noise_sd=0.02, noise_rho=0.3, signs=(-1, -1, 1),
    budget=((1, 1.0), (2, 0.5), (9, 1.0), (0, -0.5)),
    tradeoff=(1.0, -1.0, 0.0),   # TTFT against TPOT; throughput rides on its own surface
    conflict_scale=2.0,
)

_P12 = _P10 + (
    Param("max_seq_len_to_capture", INT_LOG, 256, 8192, default=8192),
    Param("swap_space", INT_UNIFORM, 0, 16, default=4),
)

D12_FANTASY = Workload(
    name="d12-fantasy",
    params=_P12,
    clauses=_C10 + (
        # without chunked prefill the batched-token budget covers the captured length
        Clause(((5, 0),), ((2, 1), (10, -1)), 0),
        # prefix caching wants a block size of at least 16
        Clause(((6, 1),), ((3, 1),), 1),
    ),
    n_obs=256, n_cand=1 << 22, n_obj=2, acq="ehvi", n_trees=200, max_depth=14,
    n_mc=64, q=16, noise_sd=0.01, noise_rho=0.0, signs=(-1, -1),
    budget=((1, 1.0), (2, 0.5), (9, 1.0), (0, -0.5), (11, 0.3)),
    fantasy=True,
)

WORKLOADS = {w.name: w for w in (TINY, D8, D10_EI, D10_EHVI3, D12_FANTASY)}
ORDER = ("tiny", "d8-ehvi2", "d10-ei", "d10-ehvi3", "d12-fantasy")

# Master seeds: 1000+c for the benchmark, 2000+c and 3000+c for extra parity runs.
def seeds(name: str):
    c = ORDER.index(name) + 1
    return (1000 + c, 2000 + c, 3000 + c)
