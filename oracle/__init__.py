"""fp64 CPU oracle of the candidate-scoring path.

TEST INFRASTRUCTURE ONLY: imported by the tests, the smoke check and the
benchmark's CPU-baseline leg, never by the product path.
"""
from .scoot_oracle import *  # noqa: F401,F403
