"""CPU oracle for the OffQ W4A4 linear path (test infrastructure; see offq_oracle.py)."""

from .offq_oracle import *  # noqa: F401,F403
