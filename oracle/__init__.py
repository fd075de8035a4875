"""fp64 CPU oracle of the Hydra-PPO scoring path. Test infrastructure only: imported by
tests/, by the package smoke check and by the benchmark's CPU-baseline leg, never by the
CUDA library or its Python binding."""
from .hydra_oracle import *  # noqa: F401,F403
from . import hydra_oracle  # noqa: F401
