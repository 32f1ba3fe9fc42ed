"""CPU oracle for PCTree drafting rounds (test infrastructure only)."""
from . import pctree_oracle  # noqa: F401
