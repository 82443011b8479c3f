"""Oracle for CaPE proposal expansion (test infrastructure only).

Confidence-aware proposal expansion, Section 3.2 ("Confidence-aware Proposal
Expansion" and "Verification of Expanded Proposals"):

* the draft's distribution p_D(. | x_{<t+i}) at proposal position i picks
  x_{t+i} = its most probable token, with confidence p_i = max p_D;
* K_i = S(p_i), S(p) = 7, 5, 3, 1 on (0, 0.3], (0.3, 0.6], (0.6, 0.8], (0.8, 1];
* the expansion set X_i holds the K_i most probable tokens other than x_{t+i};
* the expanded proposal is linearized: the gamma proposal tokens, then the
  expansion sets appended in position order.

Section 4's ablation ("The importance of confidence scores") replaces S by a
fixed size (4); ``fixed_k`` gives that variant.

Readings where the paper is silent (each fixes an integer result exactly):
* ranking is by probability, highest first, ties to the lower token id;
  -0.0 and +0.0 are the same probability (a zero confidence is reported as +0);
* the comparison with the decimal thresholds is exact: the fp32 value of p_i
  against the real number 0.3, 0.6 or 0.8 (none of which is a binary32 value,
  so whether an interval end is open or closed never matters for fp32 input);
  p_i <= 0 falls in the first bucket, p_i > 1 in the last;
* a position's set has at most V - 1 tokens (there are no more to take);
* the tree: node 0 is x_t (the last accepted token, ``root_token``), node i
  (1 <= i <= gamma) is x_{t+i} with parent i - 1, and an expansion token of
  position i is a sibling of x_{t+i} (parent i - 1).  Its ancestor-or-self
  mask is the CaPE mask;
* the cap on verified tokens (32 in Section 4, Medusa comparison) counts the
  proposal and expansion tokens, not x_t.  When the sets overflow it, the
  expansion tokens of lowest probability are dropped first (among equal
  probabilities, later positions first, then later ranks), so each kept set
  is still the top of its position;
* unused node slots (n_nodes .. max_tokens) hold token -1 with parent 0: they
  are leaves whose token no argmax equals, so acceptance never takes them.
"""
from __future__ import annotations

from fractions import Fraction
from typing import Optional

import numpy as np

# S(p) of Section 3.2: (upper end of the interval, K) for the first three
# intervals; above 0.8 the size is 1.
_S_TABLE = ((Fraction(3, 10), 7), (Fraction(6, 10), 5), (Fraction(8, 10), 3))
_S_LAST = 1


def expansion_size(p: float) -> int:
    """S(p): 7, 5, 3, 1 on (0, 0.3], (0.3, 0.6], (0.6, 0.8], (0.8, 1],
    comparing the exact value of p with the exact thresholds."""
    x = Fraction(float(p))
    for upper, k in _S_TABLE:
        if x <= upper:
            return k
    return _S_LAST


def ranked_tokens(row: np.ndarray) -> list:
    """Token ids of one distribution, most probable first, ties to the lower id."""
    vals = [float(v) + 0.0 for v in row]      # + 0.0 turns -0.0 into +0.0
    return sorted(range(len(vals)), key=lambda t: (-vals[t], t))


def expansion_set(order: list, k: int) -> list:
    """X_i: the k best-ranked tokens other than x_{t+i} = order[0]."""
    return order[1:k + 1]


def keep_after_cap(candidates: list, room: int) -> list:
    """The expansion tokens that fit in `room` slots: the most probable ones,
    equal probabilities to the earlier position, then the earlier rank.
    candidates: (probability, position, rank, token) tuples."""
    return sorted(candidates, key=lambda c: (-c[0], c[1], c[2]))[:room]


def cape_expand(probs: np.ndarray, root_token: np.ndarray, max_tokens: int = 32,
                fixed_k: Optional[int] = None):
    """CaPE expansion of B proposals.

    probs [B, gamma, V] fp32: the draft's next-token distribution at each of
    the gamma proposal positions.  root_token [B]: x_t.  max_tokens: cap on
    proposal + expansion tokens (gamma <= max_tokens).  fixed_k: None for the
    confidence-aware S(p_i), else the fixed set size.

    Returns (draft_tokens [B, 1+max_tokens] int32, parent_idx [B, 1+max_tokens]
    int32, n_nodes [B] int32, conf [B, gamma] fp32 = p_i, k_used [B, gamma]
    int32 = set sizes after the cap).
    """
    B, gamma, V = probs.shape
    assert gamma <= max_tokens
    n_out = 1 + max_tokens
    tokens = np.full((B, n_out), -1, dtype=np.int32)
    parent = np.zeros((B, n_out), dtype=np.int32)
    n_nodes = np.zeros(B, dtype=np.int32)
    conf = np.zeros((B, gamma), dtype=np.float32)
    k_used = np.zeros((B, gamma), dtype=np.int32)
    for b in range(B):
        spine = []
        candidates = []                      # (probability, position, rank, token)
        for i in range(1, gamma + 1):
            row = probs[b, i - 1]
            order = ranked_tokens(row)
            x = order[0]
            p = row[x]
            spine.append(x)
            conf[b, i - 1] = float(p) + 0.0           # a zero confidence is +0
            k = expansion_size(p) if fixed_k is None else fixed_k
            k = min(k, V - 1)
            for r, tok in enumerate(expansion_set(order, k), start=1):
                candidates.append((float(row[tok]) + 0.0, i, r, tok))
        kept = sorted(keep_after_cap(candidates, max_tokens - gamma),
                      key=lambda c: (c[1], c[2]))                 # linearized order
        tokens[b, 0] = root_token[b]
        parent[b, 0] = -1
        for i, x in enumerate(spine, start=1):
            tokens[b, i] = x
            parent[b, i] = i - 1
        node = gamma + 1
        for _, i, _, tok in kept:
            tokens[b, node] = tok
            parent[b, node] = i - 1
            k_used[b, i - 1] += 1
            node += 1
        n_nodes[b] = node
    return tokens, parent, n_nodes, conf, k_used
