"""Oracle for speculative-sampling acceptance (test infrastructure only).

Section 2 names the two acceptance strategies of speculative decoding; the
paper's GliDe-only experiments (Section 4.1, gamma = 5) use speculative
sampling, whose outputs are distributed as the target model's own samples,
with per-token acceptance rate sum_x min(p_T(x), p_D(x)) (Section 4.1,
"Metrics").  The rule, for a chain proposal x_1..x_gamma drawn from the draft's
distributions p_D,1..p_D,gamma, the target's distributions p_T,1..p_T,gamma+1
and uniform numbers u_1..u_gamma, v in [0, 1):

* position i accepts x_i when u_i * p_D,i(x_i) < p_T,i(x_i) (i.e. with
  probability min(1, p_T / p_D)); the first rejection ends the round;
* after a rejection at position i, one more token is drawn from the residual
  distribution proportional to max(0, p_T,i - p_D,i); if all gamma are
  accepted, it is drawn from p_T,gamma+1;
* a draw from weights w takes the first token whose running sum of w exceeds
  v * sum(w) (inverse-CDF sampling).

Readings where the paper is silent:
* p_T = SoftMax(target logits) at temperature 1 (random sampling), in fp64 here;
* the random numbers are inputs (uniforms [B, gamma + 1]: u_1..u_gamma, then v);
* the comparison is strict (u * p_D < p_T), so a token the target gives
  probability 0 is always rejected, and one the draft gave 0 but the target
  not is always accepted;
* if the residual weights sum to 0 (possible only through rounding) the draw
  falls back to p_T,i; if v * sum(w) reaches the total through rounding, the
  last token of positive weight is taken.
"""
from __future__ import annotations

import numpy as np


def softmax64(logits: np.ndarray) -> np.ndarray:
    z = logits.astype(np.float64)
    e = np.exp(z - z.max())
    return e / e.sum()


def inverse_cdf(w: np.ndarray, v: float) -> int:
    """First index whose running sum of w exceeds v * sum(w)."""
    total = w.sum()
    c = np.cumsum(w)
    idx = int(np.searchsorted(c, float(v) * total, side="right"))
    if idx >= len(w):
        idx = int(np.nonzero(w > 0)[0][-1])
    return idx


def accepts(u: float, p_draft: float, p_target: float) -> bool:
    """Position test: accept when u * p_D(x) < p_T(x)."""
    return float(u) * float(p_draft) < float(p_target)


def residual_weights(p_target: np.ndarray, p_draft: np.ndarray) -> np.ndarray:
    """max(0, p_T - p_D); p_T itself if that sums to 0."""
    w = np.maximum(0.0, p_target - p_draft.astype(np.float64))
    return w if w.sum() > 0 else p_target


def spec_sample_accept(draft_tokens: np.ndarray, draft_probs: np.ndarray, target_logits: np.ndarray,
                       uniforms: np.ndarray):
    """draft_tokens [B, gamma] int, draft_probs [B, gamma, V] fp32, target_logits
    [B, gamma + 1, V] fp32, uniforms [B, gamma + 1] fp32 in [0, 1).
    Returns (n_accepted [B] int32, next_token [B] int32)."""
    B, gamma = draft_tokens.shape
    n_acc = np.zeros(B, dtype=np.int32)
    nxt = np.zeros(B, dtype=np.int32)
    for b in range(B):
        n = gamma
        for i in range(gamma):
            pT = softmax64(target_logits[b, i])
            x = int(draft_tokens[b, i])
            if not accepts(uniforms[b, i], draft_probs[b, i, x], pT[x]):
                n = i
                break
        n_acc[b] = n
        if n < gamma:
            w = residual_weights(softmax64(target_logits[b, n]), draft_probs[b, n])
        else:
            w = softmax64(target_logits[b, gamma])
        nxt[b] = inverse_cdf(w, uniforms[b, gamma])
    return n_acc, nxt
