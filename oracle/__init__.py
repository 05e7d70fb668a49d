"""fp64 CPU oracle (test infrastructure only; never on the product path)."""
from . import ultratex_oracle  # noqa: F401
from .ultratex_oracle import *  # noqa: F401,F403
