"""Oracle for greedy tree acceptance (test infrastructure only).

Speculative decoding's greedy acceptance (Section 2): a proposed token is kept
iff it is the token the target would have produced greedily at that point, the
kept tokens are the longest such run, and the target's own next token after
the last kept one comes for free.  With CaPE's expanded proposal (Section 3.2)
the proposal is a token tree and "longest run" becomes the deepest node whose
whole root path is reproduced.

Conventions (readings where the paper is silent):
* node 0 is x_t, the last token already accepted; its own token is not checked;
* a_i = argmax_v logits[i, v], the lowest v among equal maxima;
* node c (parent p) matches iff draft[c] == a_p; it is accepted iff it and all
  of its ancestors except the root match;
* the result is the accepted node of greatest depth, the lowest node index
  among equals; len = its depth, path = root..node, bonus = a_node.
"""
from __future__ import annotations

import numpy as np


def row_argmax(logits: np.ndarray) -> np.ndarray:
    """First index of the maximum of each row of [..., V] fp32 logits."""
    return np.argmax(logits, axis=-1).astype(np.int32)


def tree_accept(draft_tokens: np.ndarray, parent_idx: np.ndarray, target_logits: np.ndarray):
    """Greedy acceptance for each of B trees.

    draft_tokens [B, n] int, parent_idx [B, n] int (node 0 the root, parents
    earlier than children), target_logits [B, n, V] fp32.
    Returns (path [B, n] int32 root-first and -1 padded, len [B] int32,
    bonus [B] int32).
    """
    B, n = draft_tokens.shape
    path = np.full((B, n), -1, dtype=np.int32)
    length = np.zeros(B, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    for b in range(B):
        a = row_argmax(target_logits[b])
        par = parent_idx[b]
        accepted = [False] * n
        depth = [0] * n
        accepted[0] = True
        for c in range(1, n):                     # parents precede children
            p = int(par[c])
            depth[c] = depth[p] + 1
            accepted[c] = accepted[p] and int(draft_tokens[b, c]) == int(a[p])
        best = 0
        for c in range(1, n):
            if accepted[c] and depth[c] > depth[best]:
                best = c
        chain = []
        j = best
        while j >= 0:
            chain.append(j)
            j = int(par[j]) if j != 0 else -1
        chain.reverse()
        path[b, :len(chain)] = chain
        length[b] = depth[best]
        bonus[b] = a[best]
    return path, length, bonus
