"""CPU fp64 oracle for SWAN (test infrastructure; never imported by the library)."""
from .swan_oracle import *  # noqa: F401,F403
from . import basis_oracle  # noqa: F401
