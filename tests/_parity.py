"""Parity rules between the CUDA path and the CPU oracle (see oracle/parity.py)."""
from oracle.parity import TOL, check_rows, near_tie, to_np  # noqa: F401
