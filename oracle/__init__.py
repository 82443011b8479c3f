"""CPU oracle for the GliDe-with-CaPE hot path (arXiv 2402.02082).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this
package: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py`` use it.  It shares no code with the CUDA library.

It is a plain, slow, fp64 restatement of what the path computes:

* ``attention.cross_attn``       -- GliDe cross-attention of a draft query over
  the target's cached keys/values (Section 3.1, the hd_j equation; no mask at
  inference).
* ``attention.tree_verify_attn`` -- the target's parallel verification of the
  linearized expanded proposal under the ancestor-or-self mask, of which the
  CaPE mask (Section 3.2) is the special case for CaPE's trees.
* ``attention.block_cross_attn`` -- the draft's cross-attention at training
  time under the block-wise mask (Section 3.1): every position's query over
  the target's cache of the blocks before its own.
* ``accept.tree_accept``         -- greedy acceptance (speculative decoding,
  Section 2) on a token tree: the deepest node whose root path the target's
  argmax reproduces, plus the free bonus token.
* ``cape.cape_expand``           -- CaPE's confidence-aware proposal expansion
  (Section 3.2; the fixed-size variant of Section 4): proposal tokens, S(p_i)
  sized expansion sets, and the linearized token tree.
* ``kvcache.kv_compact``         -- the cache update after verification
  (Section 3.1): the accepted path's entries become contiguous rows.
* ``sampling.spec_sample_accept`` -- speculative-sampling acceptance of a
  chain proposal (the strategy Section 2 names and Section 4.1 uses for GliDe
  alone), with the random numbers as inputs.

Every function here is pinned by tests in ``tests/test_oracle.py`` against
closed forms, library routines, brute force and invariants; none is marked
"parity unpinned".
"""
from .attention import (ancestors_or_self, block_cross_attn, block_mask, cape_mask, cross_attn,
                        tree_allowed_mask, tree_verify_attn, widen)
from .accept import row_argmax, tree_accept
from .cape import cape_expand, expansion_size
from .kvcache import kv_compact
from .sampling import spec_sample_accept

__all__ = ["ancestors_or_self", "block_cross_attn", "block_mask", "cape_mask", "cross_attn", "tree_allowed_mask",
           "tree_verify_attn", "widen", "row_argmax", "tree_accept", "cape_expand", "expansion_size", "kv_compact",
           "spec_sample_accept"]
