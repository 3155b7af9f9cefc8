"""CPU oracle for the VarRate hot path: test infrastructure only (see varrate_oracle)."""
from .varrate_oracle import *  # noqa: F401,F403
from . import varrate_oracle as vo  # noqa: F401
