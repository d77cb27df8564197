"""Float64 CPU oracle of the fuse-and-verify step (test infrastructure only)."""
from .asymspec_oracle import *  # noqa: F401,F403
