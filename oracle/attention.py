"""fp64 oracle for the two KV-cache attention steps (test infrastructure only).

Notation follows the paper: per target layer and head j, the cached keys and
values K^{l,j}, V^{l,j} (Section 3.1); the draft query Q^{m,j}; scale
1/sqrt(d_k).  Tensor layouts are those of the library boundary:

    queries  [B, nq, H, D]
    K, V     [B, H_kv, S_cap, D] (rows >= kv_len[b] + n are unused capacity)
    kv_len   [B]
    parent   [B, n]  (-1 for a root, else an earlier node)

bf16 inputs arrive as uint16 bit patterns and are widened exactly; fp32 inputs
are widened exactly.  All arithmetic is fp64.
"""
from __future__ import annotations

from typing import Iterable, Optional, Sequence, Tuple

import numpy as np


def widen(x: np.ndarray) -> np.ndarray:
    """Exact value of a bf16 (uint16 bit pattern) or fp32 array, as fp64."""
    if x.dtype == np.uint16:
        return (x.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    if x.dtype in (np.float32, np.float64):
        return x.astype(np.float64)
    raise TypeError(f"unsupported dtype {x.dtype}")


def _softmax_rows_attend(scores: np.ndarray, allowed: np.ndarray, values: np.ndarray) -> np.ndarray:
    """Row-wise SoftMax over the allowed entries of `scores`, times `values`.

    scores [r, k], allowed [r, k] bool, values [k, D] -> [r, D].  Disallowed
    entries are -inf before the softmax (the paper's mask convention).  A row
    with no allowed entry has an empty softmax, which the paper leaves
    undefined; it yields zeros here.
    """
    s = np.where(allowed, scores, -np.inf)
    out = np.zeros((s.shape[0], values.shape[1]), dtype=np.float64)
    for r in range(s.shape[0]):
        if not allowed[r].any():
            continue
        m = s[r].max()
        e = np.exp(s[r] - m)          # exp(-inf) = 0 for masked keys
        out[r] = (e @ values) / e.sum()
    return out


def kv_head(h: int, H: int, H_kv: int) -> int:
    """The cached key/value head that query head h reads.  H_kv = H is plain
    multi-head attention; with fewer cached heads (grouped-query attention, as
    in Mistral-7B: 32 query heads over 8 key/value heads) each run of H / H_kv
    consecutive query heads shares one cached head."""
    if H % H_kv:
        raise ValueError("the query heads must split evenly over the key/value heads")
    return h // (H // H_kv)


def _pairs(B: int, H: int, pairs: Optional[Iterable[Tuple[int, int]]]):
    if pairs is None:
        return [(b, h) for b in range(B) for h in range(H)]
    return list(pairs)


def cross_attn(q_draft: np.ndarray, K: np.ndarray, V: np.ndarray, kv_len: Sequence[int],
               scale: Optional[float] = None, pairs=None) -> np.ndarray:
    """GliDe cross-attention, Section 3.1:

        hd_j = SoftMax(Q^{m,j} (K^{l,j})^T / sqrt(d_k)) V^{l,j}

    over every cached prefix key 0..kv_len[b]-1 (no mask at inference: the
    block-wise mask is a training-only device).  q_draft [B, nq, H, D] ->
    out [B, nq, H, D].  `pairs` restricts the work to some (b, h); the other
    outputs are NaN.
    """
    B, nq, H, D = q_draft.shape
    sc = 1.0 / np.sqrt(D) if not scale else float(scale)
    out = np.full((B, nq, H, D), np.nan)
    for b, h in _pairs(B, H, pairs):
        L = int(kv_len[b])
        hk = kv_head(h, H, K.shape[1])
        Kb = widen(K[b, hk, :L])
        Vb = widen(V[b, hk, :L])
        Q = widen(q_draft[b, :, h, :])                  # [nq, D]
        scores = (Q @ Kb.T) * sc                        # Q K^T / sqrt(d_k)
        allowed = np.ones_like(scores, dtype=bool)
        out[b, :, h, :] = _softmax_rows_attend(scores, allowed, Vb)
    return out


def ancestors_or_self(parent: Sequence[int], i: int) -> list:
    """Node i and every node on its path to the root, following parent links."""
    chain = []
    j = int(i)
    while j >= 0:
        chain.append(j)
        j = int(parent[j])
    return chain


def tree_allowed_mask(parent: Sequence[int], kv_len: int) -> np.ndarray:
    """[n, kv_len + n] bool: which keys each tree query may attend to.

    Every cached prefix key is visible to every query.  Tree key kv_len + j is
    visible to query i iff j is i or an ancestor of i (the token-tree verifier
    the paper borrows for CaPE, Section 3.2).
    """
    n = len(parent)
    allowed = np.zeros((n, kv_len + n), dtype=bool)
    allowed[:, :kv_len] = True
    for i in range(n):
        for j in ancestors_or_self(parent, i):
            allowed[i, kv_len + j] = True
    return allowed


def tree_verify_attn(q_tree: np.ndarray, parent_idx: np.ndarray, K: np.ndarray, V: np.ndarray,
                     kv_len: Sequence[int], scale: Optional[float] = None, pairs=None) -> np.ndarray:
    """Target verification of the linearized tree, Section 3.2.

    The n tree tokens' own keys/values sit at cache rows kv_len[b] .. kv_len[b]+n-1
    in linearized order.  Query i attends to all prefix keys and to the tree
    keys of its ancestors and itself:

        o_i = SoftMax(mask(q_i K^T / sqrt(d_k))) V

    q_tree [B, n, H, D] -> out [B, n, H, D].
    """
    B, n, H, D = q_tree.shape
    sc = 1.0 / np.sqrt(D) if not scale else float(scale)
    out = np.full((B, n, H, D), np.nan)
    masks = {}
    for b, h in _pairs(B, H, pairs):
        L = int(kv_len[b])
        if b not in masks:
            masks[b] = tree_allowed_mask(parent_idx[b], L)
        hk = kv_head(h, H, K.shape[1])
        Kb = widen(K[b, hk, :L + n])
        Vb = widen(V[b, hk, :L + n])
        Q = widen(q_tree[b, :, h, :])
        scores = (Q @ Kb.T) * sc
        out[b, :, h, :] = _softmax_rows_attend(scores, masks[b], Vb)
    return out


def cape_mask(gamma: int, pos: Sequence[int]) -> np.ndarray:
    """The CaPE verification mask over the linearized proposal P (Section 3.2).

    P = (x_{t+1}, ..., x_{t+beta}), 1-indexed; the first gamma entries are the
    proposal, pos(i) is the position an expansion token stands for (pos(i) = i
    on the proposal).  Entry (i, j) is kept iff (j <= gamma and pos(i) > j) or
    i = j.  `pos` is indexed by tree node (pos[0] is the root x_t and is
    ignored).  Returns the beta x beta keep-matrix, 0-indexed.
    """
    beta = len(pos) - 1
    keep = np.zeros((beta, beta), dtype=bool)
    for i in range(1, beta + 1):
        for j in range(1, beta + 1):
            if (j <= gamma and pos[i] > j) or i == j:
                keep[i - 1, j - 1] = True
    return keep


def block_mask(T: int, L: int) -> np.ndarray:
    """The training-time block-wise mask of the draft's cross-attention
    (Section 3.1, "Block-wise Attention Mask"), as printed: entry (j, k) of the
    T x T attention matrix is kept iff block(j) > block(k), block(x) = the index
    of x's block of L tokens."""
    block = np.arange(T) // L
    return block[:, None] > block[None, :]


def block_cross_attn(q: np.ndarray, K: np.ndarray, V: np.ndarray, seq_len: Sequence[int], L: int,
                     scale: Optional[float] = None, pairs=None) -> np.ndarray:
    """The draft's cross-attention at training time (Section 3.1): the query of
    every position j of a training sequence attends to the target's keys and
    values of the positions k with block(j) > block(k) (the blocks of L tokens
    before j's own block), so that training sees the delayed cache that
    speculation sees.  q [B, T, H, D]; K, V [B, H_kv, S_cap, D] hold the
    target's keys/values of positions 0..T-1; seq_len [B] tokens of each
    sequence.  A position with nothing to attend to (the first block) and a
    position at or past seq_len get zeros.  -> out [B, T, H, D]."""
    B, T, H, D = q.shape
    sc = 1.0 / np.sqrt(D) if not scale else float(scale)
    out = np.zeros((B, T, H, D), dtype=np.float64)
    for b, h in _pairs(B, H, pairs):
        n = int(seq_len[b])
        if n == 0:
            continue
        hk = kv_head(h, H, K.shape[1])
        allowed = block_mask(n, L)
        Kb = widen(K[b, hk, :n])
        Vb = widen(V[b, hk, :n])
        Q = widen(q[b, :n, h, :])
        out[b, :n, h, :] = _softmax_rows_attend((Q @ Kb.T) * sc, allowed, Vb)
    return out
