"""CPU oracle for the ALTR reduction path -- test infrastructure only.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference arms may import this package.  The product path never does.
"""
from .altr import (NEAR_TIE, budget_from_ratio, budget_split, consistency, exact_r, exact_sigma,
                   pick_positions, renyi2_entropy, select_image, stride)

__all__ = ["NEAR_TIE", "budget_from_ratio", "budget_split", "consistency", "exact_r", "exact_sigma",
           "pick_positions", "renyi2_entropy", "select_image", "stride"]
