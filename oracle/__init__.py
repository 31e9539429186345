"""fp64 CPU oracle (test infrastructure only; see hdf_oracle's header)."""
from .hdf_oracle import *  # noqa: F401,F403
