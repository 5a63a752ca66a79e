"""Float64 CPU oracle for the draft-tree verification pass.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
execute this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code, headers, tables or helpers with the CUDA library under
``paper_2502_11018_gb300/csrc``; the only thing both sides consume is the
seeded input generator module ``paper_2502_11018_gb300.inputs``, which holds
none of the method's arithmetic.

What it computes (GRIFFIN, arXiv 2502.11018):

* the draft-and-verify cycle of Section 3: one target forward over all draft
  tokens, then acceptance of a subset (``tree``, ``attention``, ``lmhead``,
  ``accept``, ``compact``);
* the draft tree of Appendix C (dynamic tree, 60 draft tokens, depth 6),
  encoded as a parent-index array with nodes in topological order;
* the rule of Section 4.1 that rejecting a draft token discards every later
  token of its draft sequence (the whole subtree);
* losslessness (Section 5): greedy acceptance reproduces greedy decoding, and
  temperature-1 acceptance reproduces the target distribution;
* the token-alignable training objective of the draft model (Section 4.1,
  Eqs. 2-5 and the loss of the Implementation Details appendix: top-k
  predictable masks, chain alignment masks, masked per-sequence loss) in
  ``tat``;
* the target model's decoder layers around the tree attention (RMSNorm,
  projections, SwiGLU MLP, residuals) in ``layer``;
* the draft model's Token-Guided Fusion module (Eqs. 6-8) in ``tgf``;
* the dynamic draft tree built from top-k expansions and a rerank (the draft
  side of a cycle) in ``draft_tree``.

Every function works in float64 with plain loops or single library
primitives (a matmul, a sort), in the order the definition states.

Parity pins: every function here is pinned by a ``-m "not gpu"`` test in
``tests/test_oracle_*.py`` against something other than itself (brute force,
closed forms, textbook special cases, statistical losslessness).  No function
is "parity unpinned".
"""

from .tree import tree_build, GV_OK, GV_ERR_INVALID_TREE, GV_ERR_CAPACITY  # noqa: F401
from .attention import rope_rotate, tree_attention  # noqa: F401
from .lmhead import lmhead_logits, select_argmax, select_topk, row_logsumexp  # noqa: F401
from .accept import accept_greedy, accept_sampling  # noqa: F401
from .compact import kv_compact  # noqa: F401
from .step import verify_step  # noqa: F401
from .tat import predictable_mask, alignment_mask, token_loss, feature_loss, tat_pass  # noqa: F401
from .layer import rmsnorm, linear, silu, swiglu, decoder_layer  # noqa: F401
from .tgf import layernorm, tgf_forward  # noqa: F401
from .draft_tree import draft_tree, pool_size  # noqa: F401
