"""Oracle for the KV-cache update after verification (test infrastructure only).

Section 3.1 (how the draft reuses the target's KV cache): after a
verification step the target keeps the cache entries of the tokens it
accepted and discards those of the rejected ones.  With the linearized tree
of Section 3.2 written at rows kv_len[b] .. kv_len[b]+n-1 (node j at row
kv_len[b]+j), "keep" means: the entries of the accepted root path
path[b, 0..len[b]] (node 0 = x_t, then the accepted proposal tokens) become
the contiguous rows kv_len[b] .. kv_len[b]+len[b], in path order, and the
cache length grows to kv_len[b] + len[b] + 1.  The new bonus token has no
entry yet: it is node 0 of the next round's tree.

Rows outside the written range keep their old contents.
"""
from __future__ import annotations

import numpy as np


def kv_compact(K: np.ndarray, V: np.ndarray, kv_len, path: np.ndarray, length):
    """K, V [..., B, H, S_cap, D] (any leading layer dimensions; any dtype),
    kv_len [B], path [B, n] (root-first node indices, -1 padded), length [B].
    Returns (K', V', new_kv_len [B] int32); the inputs are not modified."""
    K2 = K.copy()
    V2 = V.copy()
    B = len(kv_len)
    new_len = np.zeros(B, dtype=np.int32)
    for b in range(B):
        L = int(kv_len[b])
        m = int(length[b]) + 1
        src = [L + int(path[b, k]) for k in range(m)]
        K2[..., b, :, L:L + m, :] = K[..., b, :, :, :][..., src, :]
        V2[..., b, :, L:L + m, :] = V[..., b, :, :, :][..., src, :]
        new_len[b] = L + m
    return K2, V2, new_len
