"""ALTR visual-token reduction (arxiv 2607.13500) on GB300.

Per token, the second-order Renyi entropy of the channel-magnitude
distribution (importance, Eq. 3-4) and the cosine between the vision
encoder's final-layer MLP input and output (consistency, Eq. 6); per image,
the K1 most important tokens plus K2 tokens at a stride along the rest sorted
by consistency (Algorithm 1), gathered into a compact [sum K, D] tensor.

The work runs in libtr.so (hand-written CUDA for sm_103a, C ABI in
include/tr.h); this package is its Python binding.  ``mlp`` runs the vision
encoder's final-layer MLP (Eq. 5) on the tensor cores with the scoring fused
into its second GEMM, for callers that own that MLP; ``project_kept`` runs the
projector's first layer on the kept tokens, reading them from x by index, and
``project`` the same layer on the gathered rows y (the faster route).
"""
from .api import (Mlp, MlpResult, Pipeline, Reducer, ReduceResult, budgets, mlp, project, project_kept, reduce,
                  score, select, workspace_bytes)

__all__ = ["Mlp", "MlpResult", "Pipeline", "Reducer", "ReduceResult", "budgets", "mlp", "project", "project_kept",
           "reduce", "score", "select", "workspace_bytes"]
