"""Seeded synthetic inputs for the GliDe/CaPE attention and acceptance path.

This module only draws random numbers and lays them out. It holds none of the
method's arithmetic (no attention, no masking, no argmax, no tree walk), so the
CPU oracle and the CUDA path can both consume its arrays without sharing any
computation.

Shapes follow the target models of the paper's experiments (Section 4.1:
Vicuna-7B/13B/33B, head dim 128, vocabulary 32000).  The tree recipe follows
the CaPE verification setting (Section 3.2): node 0 is the last accepted token
x_t, every other node has a parent with a smaller index, and sibling tokens are
distinct (an expansion set never repeats the proposal token at its position).

All floating-point tensors are returned as numpy arrays: bf16 as ``uint16``
bit patterns (round-to-nearest-even from fp32) and fp32 as ``float32``.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np

BF16_NAN = np.uint16(0x7FC0)


# --------------------------------------------------------------------------
# number formats
# --------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest, ties to even); finite input."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(u: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32 (used for host-side display only)."""
    return (np.ascontiguousarray(u, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _rng(seed: int, *stream: int) -> np.random.Generator:
    """Independent generator per (seed, stream) so tensors do not depend on draw order."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *stream])))


def normal_values(seed: int, stream: int, shape: Sequence[int], dtype: str, std: float = 1.0) -> np.ndarray:
    g = _rng(seed, stream)
    x = g.standard_normal(size=tuple(shape), dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    if dtype == "f32":
        return x
    raise ValueError(dtype)


# --------------------------------------------------------------------------
# trees (parent arrays in linearized order, node 0 = root x_t)
# --------------------------------------------------------------------------
def chain_tree(n: int) -> np.ndarray:
    """Plain speculative-decoding proposal: x_t -> x_{t+1} -> ... (a chain)."""
    return np.arange(-1, n - 1, dtype=np.int32)


def random_tree(seed: int, n: int, max_depth: int, max_branch: int) -> np.ndarray:
    """Grow a tree to n nodes: repeatedly pick, uniformly, an existing node with
    depth < max_depth and fewer than max_branch children, and give it a child."""
    g = _rng(seed, 7)
    parent = np.full(n, -1, dtype=np.int32)
    depth = np.zeros(n, dtype=np.int64)
    nchild = np.zeros(n, dtype=np.int64)
    for i in range(1, n):
        cands = [j for j in range(i) if depth[j] < max_depth and nchild[j] < max_branch]
        if not cands:
            raise ValueError("tree shape limits too tight for n nodes")
        p = cands[int(g.integers(len(cands)))]
        parent[i] = p
        depth[i] = depth[p] + 1
        nchild[p] += 1
    return parent


def cape_tree(expansion_sizes: Sequence[int]) -> tuple:
    """Linearized CaPE expanded proposal as a parent array.

    Node 0 is x_t; nodes 1..gamma are the proposal x_{t+1}..x_{t+gamma}; the
    expansion tokens of position j (|X_j| = expansion_sizes[j-1]) follow, in
    position order.  Returns (parent, pos) where pos[i] is the paper's pos()
    for node i >= 1 (pos[i] = i on the proposal) and pos[0] = 0.
    """
    gamma = len(expansion_sizes)
    parent = [-1] + [i - 1 for i in range(1, gamma + 1)]
    pos = [0] + list(range(1, gamma + 1))
    for j, k in enumerate(expansion_sizes, start=1):
        for _ in range(k):
            parent.append(j - 1)
            pos.append(j)
    return np.asarray(parent, dtype=np.int32), np.asarray(pos, dtype=np.int32)


def tree_depths(parent: np.ndarray) -> np.ndarray:
    d = np.zeros(len(parent), dtype=np.int64)
    for i in range(1, len(parent)):
        d[i] = d[parent[i]] + 1 if parent[i] >= 0 else 0
    return d


# --------------------------------------------------------------------------
# tokens and logits for acceptance
# --------------------------------------------------------------------------
def draft_tokens(seed: int, parent: np.ndarray, vocab: int) -> np.ndarray:
    """Draft token of every node; siblings get distinct tokens."""
    g = _rng(seed, 11)
    n = len(parent)
    tok = np.zeros(n, dtype=np.int32)
    tok[0] = int(g.integers(vocab))
    for p in range(n):
        kids = [c for c in range(n) if parent[c] == p]
        if kids:
            tok[kids] = g.choice(vocab, size=len(kids), replace=False)
    return tok


def planted_logits(seed: int, parent: np.ndarray, tokens: np.ndarray, vocab: int,
                   std: float, p_accept: float) -> np.ndarray:
    """fp32 logits [n, vocab] ~ N(0, std).  For a node with children, with
    probability p_accept one child's token is made the unique row maximum
    (row max + 1); otherwise a token that is no child's gets that value."""
    g = _rng(seed, 13)
    n = len(parent)
    lg = g.standard_normal(size=(n, vocab), dtype=np.float32) * np.float32(std)
    for p in range(n):
        kids = [c for c in range(n) if parent[c] == p]
        if not kids:
            continue
        top = np.float32(lg[p].max() + np.float32(1.0))
        if g.random() < p_accept:
            c = kids[int(g.integers(len(kids)))]
            lg[p, tokens[c]] = top
        else:
            taken = set(int(tokens[c]) for c in kids)
            while True:
                t = int(g.integers(vocab))
                if t not in taken:
                    break
            lg[p, t] = top
    return lg


def draft_probs(seed: int, B: int, gamma: int, vocab: int, quantum: float = 0.0) -> np.ndarray:
    """fp32 draft distributions [B, gamma, vocab] for proposal expansion.

    Each row's largest entry (the confidence) is drawn uniformly from
    [0.05, 0.98], so the four confidence bands of CaPE's size rule are all
    visited; the remaining mass is spread over the other tokens with a
    heavy-tailed (Gamma(0.3)) profile, as an LLM's next-token distribution
    has a few runners-up and a long flat tail.  With quantum > 0 every entry
    is rounded to a multiple of it, which creates many exact ties (and zeros).
    """
    g = _rng(seed, 31)
    out = np.empty((B, gamma, vocab), dtype=np.float32)
    for b in range(B):
        for i in range(gamma):
            conf = g.uniform(0.05, 0.98)
            tail = g.gamma(0.3, size=vocab - 1)
            if vocab > 1:
                tail *= (1.0 - conf) / tail.sum()
            tail = np.minimum(tail, conf)
            row = np.insert(tail, int(g.integers(vocab)), conf)
            if quantum > 0:
                row = np.round(row / quantum) * quantum
            out[b, i] = row
    return out


def root_tokens(seed: int, B: int, vocab: int) -> np.ndarray:
    """x_t of each sequence (the token the next tree hangs from)."""
    return _rng(seed, 32).integers(vocab, size=B).astype(np.int32)


def sample_tokens(seed: int, probs: np.ndarray) -> np.ndarray:
    """One token drawn from each distribution of probs [..., V] (the draft
    model's own sampling of its proposal)."""
    g = _rng(seed, 33)
    flat = probs.reshape(-1, probs.shape[-1]).astype(np.float64)
    out = np.array([g.choice(flat.shape[1], p=row / row.sum()) for row in flat], dtype=np.int32)
    return out.reshape(probs.shape[:-1])


def target_logits_near(seed: int, draft_probs: np.ndarray, mix: float, extra_rows: int = 1) -> np.ndarray:
    """fp32 target logits [B, gamma + extra_rows, V] whose distributions mix the
    draft's (weight `mix`) with independent heavy-tailed ones, so that a
    proposal is accepted part of the time; the extra rows are independent."""
    g = _rng(seed, 34)
    B, gamma, V = draft_probs.shape
    other = g.gamma(0.3, size=(B, gamma + extra_rows, V))
    other /= other.sum(-1, keepdims=True)
    p = other.copy()
    p[:, :gamma] = mix * draft_probs.astype(np.float64) + (1.0 - mix) * other[:, :gamma]
    return np.log(np.maximum(p, 1e-30)).astype(np.float32)


def uniforms(seed: int, shape) -> np.ndarray:
    """fp32 uniform numbers in [0, 1) (the random numbers a sampling step draws)."""
    u = _rng(seed, 35).random(size=tuple(shape)).astype(np.float32)
    return np.minimum(u, np.float32(0.99999994))


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    D: int
    dtype: str            # "bf16" or "f32"
    kv_len: tuple         # per-sequence prefix length (len B)
    n: int                # tree nodes per sequence
    tree: str             # "chain" or "random"
    max_depth: int
    max_branch: int
    gamma: int            # sequential 1-query draft steps per round
    vocab: int
    logit_std: float
    p_accept: float
    seed: int

    @property
    def S_cap(self) -> int:
        need = max(self.kv_len) + self.n
        return (need + 15) // 16 * 16

    @property
    def max_kv_len(self) -> int:
        return max(self.kv_len)


def _ragged(seed: int, B: int, lo: int, hi: int) -> tuple:
    g = _rng(seed, 3)
    return tuple(int(x) for x in g.integers(lo, hi + 1, size=B))


def workloads() -> List[Workload]:
    """The five evaluation shapes: a tiny fp32 case and four Vicuna-shaped bf16 layers."""
    return [
        Workload("tiny-f32", B=1, H=4, D=64, dtype="f32", kv_len=(128,), n=5, tree="chain",
                 max_depth=4, max_branch=1, gamma=1, vocab=1000, logit_std=2.0, p_accept=0.7, seed=1000),
        Workload("vicuna7b-chain", B=1, H=32, D=128, dtype="bf16", kv_len=(2048,), n=6, tree="chain",
                 max_depth=5, max_branch=1, gamma=5, vocab=32000, logit_std=1.0, p_accept=0.7, seed=1001),
        Workload("vicuna7b-cape-tree", B=1, H=32, D=128, dtype="bf16", kv_len=(4096,), n=26, tree="random",
                 max_depth=5, max_branch=4, gamma=1, vocab=32000, logit_std=1.0, p_accept=0.7, seed=1002),
        Workload("vicuna13b-ragged-b8", B=8, H=40, D=128, dtype="bf16", kv_len=_ragged(1003, 8, 512, 4096),
                 n=26, tree="random", max_depth=5, max_branch=4, gamma=1, vocab=32000, logit_std=1.0,
                 p_accept=0.7, seed=1003),
        Workload("vicuna33b-long-b4", B=4, H=52, D=128, dtype="bf16", kv_len=(16384,) * 4, n=64, tree="random",
                 max_depth=6, max_branch=6, gamma=5, vocab=32000, logit_std=1.0, p_accept=0.6, seed=1004),
    ]


def workload(name: str) -> Workload:
    for w in workloads():
        if w.name == name:
            return w
    raise KeyError(name)


def make_trees(w: Workload) -> np.ndarray:
    if w.tree == "chain":
        return np.stack([chain_tree(w.n) for _ in range(w.B)])
    return np.stack([random_tree(w.seed * 131 + b, w.n, w.max_depth, w.max_branch) for b in range(w.B)])


def fill_kv(w: Workload, which: int, out: Optional[np.ndarray] = None, garbage: str = "nan") -> np.ndarray:
    """K (which=0) or V (which=1) cache [B, H, S_cap, D].  Rows below
    kv_len[b] + n hold N(0,1) values; rows above hold `garbage` ("nan" or
    "zero"), standing in for unused cache capacity."""
    shape = (w.B, w.H, w.S_cap, w.D)
    if out is None:
        out = np.empty(shape, dtype=np.uint16 if w.dtype == "bf16" else np.float32)
    for b in range(w.B):
        rows = w.kv_len[b] + w.n
        for h in range(w.H):
            out[b, h, :rows] = normal_values(w.seed * 7919 + b * 1009 + h, 100 + which, (rows, w.D), w.dtype)
            if garbage == "nan":
                out[b, h, rows:] = BF16_NAN if w.dtype == "bf16" else np.float32(np.nan)
            else:
                out[b, h, rows:] = 0
    return out


def make_queries(w: Workload) -> Dict[str, np.ndarray]:
    """gamma draft queries [gamma, B, 1, H, D] and tree queries [B, n, H, D]."""
    return {
        "q_draft": normal_values(w.seed, 201, (w.gamma, w.B, 1, w.H, w.D), w.dtype),
        "q_tree": normal_values(w.seed, 202, (w.B, w.n, w.H, w.D), w.dtype),
    }


def make_accept_inputs(w: Workload, parent: np.ndarray) -> Dict[str, np.ndarray]:
    tok = np.stack([draft_tokens(w.seed * 17 + b, parent[b], w.vocab) for b in range(w.B)])
    lg = np.stack([planted_logits(w.seed * 19 + b, parent[b], tok[b], w.vocab, w.logit_std, w.p_accept)
                   for b in range(w.B)])
    return {"draft_tokens": tok, "target_logits": lg}


def make_case(w: Workload, garbage: str = "nan", with_kv: bool = True) -> Dict[str, np.ndarray]:
    """Every input of one speculative round of workload w, as numpy arrays."""
    parent = make_trees(w)
    case = {"parent_idx": parent, "kv_len": np.asarray(w.kv_len, dtype=np.int32)}
    case.update(make_queries(w))
    case.update(make_accept_inputs(w, parent))
    if with_kv:
        case["K"] = fill_kv(w, 0, garbage=garbage)
        case["V"] = fill_kv(w, 1, garbage=garbage)
    return case
