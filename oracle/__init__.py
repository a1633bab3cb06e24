"""CPU oracle for the CURE repair-verify step: test infrastructure only.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg import this package; the library's product path never does.
"""
from .cure_oracle import (score_draft, row_argmax, lm_head_argmax, branch_budget, select_ufps, build_tree, anc_set,
                          cache_rows, tree_rows_in_cache, tree_attn, accept, sample_target, resync)

__all__ = ["score_draft", "row_argmax", "lm_head_argmax", "branch_budget", "select_ufps", "build_tree", "anc_set",
           "cache_rows", "tree_rows_in_cache", "tree_attn", "accept", "sample_target", "resync"]
