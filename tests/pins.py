"""Independent pins for the CPU oracle.

Each ``check_*`` takes the oracle function(s) under test as arguments and
raises AssertionError when they disagree with something the paper or plain
mathematics fixes: a closed form, a library routine the special case reduces
to, a brute-force enumeration, a hand-worked example or an invariant.  Tests
call them with the real oracle (must pass) and with mutants that carry a
planted mistake (must fail), which shows the pins can see such mistakes.
"""
from __future__ import annotations

import itertools
import math
import os

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def _randn(g, *shape):
    return g.standard_normal(shape)


# ---------------------------------------------------------------- attention
def check_single_key(cross_attn):
    """kv_len = 1: softmax over one key has weight 1, so o = V[0] exactly."""
    g = _rng(1)
    B, H, D = 2, 3, 16
    K = _randn(g, B, H, 4, D)
    V = _randn(g, B, H, 4, D)
    q = _randn(g, B, 1, H, D)
    o = cross_attn(q, K, V, [1, 1])
    assert np.array_equal(o[:, 0], V[:, :, 0, :]), "single key must return V[0]"


def check_two_keys_closed_form(cross_attn):
    """Two keys: o = sigma(s0 - s1) v0 + sigma(s1 - s0) v1 with s = q.k / sqrt(D)."""
    g = _rng(2)
    D = 8
    for _ in range(5):
        q = _randn(g, 1, 1, 1, D)
        K = _randn(g, 1, 1, 2, D)
        V = _randn(g, 1, 1, 2, D)
        s0 = float(sum(q[0, 0, 0, d] * K[0, 0, 0, d] for d in range(D))) / math.sqrt(D)
        s1 = float(sum(q[0, 0, 0, d] * K[0, 0, 1, d] for d in range(D))) / math.sqrt(D)
        w0 = 1.0 / (1.0 + math.exp(s1 - s0))
        want = w0 * V[0, 0, 0] + (1.0 - w0) * V[0, 0, 1]
        got = cross_attn(q, K, V, [2])[0, 0, 0]
        assert np.allclose(got, want, rtol=1e-13, atol=1e-13), "two-key closed form"


def check_cross_vs_sdpa(cross_attn):
    """Unmasked decode attention is torch's scaled_dot_product_attention (fp64)."""
    g = _rng(3)
    B, H, D, S = 2, 3, 32, 37
    K = _randn(g, B, H, S + 5, D)
    V = _randn(g, B, H, S + 5, D)
    q = _randn(g, B, 1, H, D)
    kv_len = [S, 11]
    o = cross_attn(q, K, V, kv_len)
    for b in range(B):
        L = kv_len[b]
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[b].transpose(1, 0, 2)),          # [H, 1, D]
            torch.from_numpy(K[b, :, :L]), torch.from_numpy(V[b, :, :L]))
        assert np.allclose(o[b, 0], ref[:, 0].numpy(), rtol=1e-12, atol=1e-12), "cross vs SDPA"


def check_chain_is_causal(tree_verify_attn):
    """A chain tree is causal attention over prefix + chain (decode with a cache)."""
    g = _rng(4)
    B, H, D, n = 2, 2, 16, 6
    kv_len = [9, 0]
    K = _randn(g, B, H, 9 + n + 3, D)
    V = _randn(g, B, H, 9 + n + 3, D)
    q = _randn(g, B, n, H, D)
    parent = np.stack([np.arange(-1, n - 1)] * B)
    o = tree_verify_attn(q, parent, K, V, kv_len)
    for b in range(B):
        L = kv_len[b]
        keep = torch.tensor([[k <= L + i for k in range(L + n)] for i in range(n)])
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[b].transpose(1, 0, 2)), torch.from_numpy(K[b, :, :L + n]),
            torch.from_numpy(V[b, :, :L + n]), attn_mask=keep)
        assert np.allclose(o[b], ref.numpy().transpose(1, 0, 2), rtol=1e-12, atol=1e-12), "chain != causal"


def check_single_node_is_decode(tree_verify_attn):
    """A one-node tree attends to the prefix plus its own key: plain decode over kv_len + 1 keys."""
    g = _rng(5)
    H, D, L = 3, 16, 20
    K = _randn(g, 1, H, L + 4, D)
    V = _randn(g, 1, H, L + 4, D)
    q = _randn(g, 1, 1, H, D)
    o = tree_verify_attn(q, np.array([[-1]]), K, V, [L])
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q[0].transpose(1, 0, 2)), torch.from_numpy(K[0, :, :L + 1]),
        torch.from_numpy(V[0, :, :L + 1]))
    assert np.allclose(o[0, 0], ref[:, 0].numpy(), rtol=1e-12, atol=1e-12), "single node != decode"


def check_uniform_keys_mean(tree_verify_attn):
    """Equal keys give equal scores, so o_i is the plain mean of V over the
    keys query i may see: every prefix key plus its ancestors and itself.
    Random V makes the mean identify exactly which rows were used."""
    g = _rng(6)
    H, D, L = 2, 8, 7
    parent = np.array([-1, 0, 0, 1, 3, 2, 1, 4])
    n = len(parent)
    k = _randn(g, D)
    K = np.broadcast_to(k, (1, H, L + n + 2, D)).copy()
    V = _randn(g, 1, H, L + n + 2, D)
    q = _randn(g, 1, n, H, D)
    o = tree_verify_attn(q, parent[None], K, V, [L])
    for i in range(n):
        anc = set()
        j = i
        while j != -1:
            anc.add(j)
            j = parent[j]
        rows = list(range(L)) + [L + j for j in sorted(anc)]
        want = V[0][:, rows].mean(axis=1)
        assert np.allclose(o[0, i], want, rtol=1e-12, atol=1e-12), f"uniform-key mean, node {i}"


def check_planted_key(cross_attn):
    """One key whose score exceeds every other by ~1000 takes all the weight:
    o = V[k*] to within exp(-900).  Also needs a max-shifted softmax (exp(1000)
    overflows fp64)."""
    g = _rng(7)
    D, L = 16, 50
    K = _randn(g, 1, 1, L, D) * 0.01
    q = _randn(g, 1, 1, 1, D)
    kstar = 17
    K[0, 0, kstar] = q[0, 0, 0] * (1000.0 * math.sqrt(D) / float(q[0, 0, 0] @ q[0, 0, 0]))
    V = _randn(g, 1, 1, L, D)
    o = cross_attn(q, K, V, [L])
    assert np.all(np.isfinite(o)), "overflow in softmax"
    assert np.allclose(o[0, 0, 0], V[0, 0, kstar], rtol=0, atol=1e-12), "planted key"


def check_prefix_permutation(tree_verify_attn):
    """Permuting the cached prefix rows (K and V together) leaves every output unchanged."""
    g = _rng(8)
    H, D, L = 2, 8, 13
    parent = np.array([-1, 0, 1, 0])
    n = len(parent)
    K = _randn(g, 1, H, L + n, D)
    V = _randn(g, 1, H, L + n, D)
    q = _randn(g, 1, n, H, D)
    o = tree_verify_attn(q, parent[None], K, V, [L])
    perm = np.concatenate([g.permutation(L), np.arange(L, L + n)])
    o2 = tree_verify_attn(q, parent[None], K[:, :, perm], V[:, :, perm], [L])
    assert np.allclose(o, o2, rtol=1e-12, atol=1e-12), "prefix permutation"


def check_tree_relabel(tree_verify_attn):
    """Renumbering the tree nodes in another topological order (parents,
    queries and tree K/V rows moved together) permutes the outputs likewise."""
    g = _rng(9)
    H, D, L = 2, 8, 5
    parent = np.array([-1, 0, 0, 1, 1, 2, 3, 2])
    n = len(parent)
    K = _randn(g, 1, H, L + n, D)
    V = _randn(g, 1, H, L + n, D)
    q = _randn(g, 1, n, H, D)
    o = tree_verify_attn(q, parent[None], K, V, [L])
    # a different topological order: breadth-first with reversed sibling order
    order = [0]
    frontier = [0]
    while frontier:
        nxt = []
        for p in frontier:
            kids = [c for c in range(n) if parent[c] == p][::-1]
            order += kids
            nxt += kids
        frontier = nxt
    new_of = {old: new for new, old in enumerate(order)}
    parent2 = np.array([-1 if parent[old] < 0 else new_of[parent[old]] for old in order])
    rows = np.concatenate([np.arange(L), L + np.array(order)])
    o2 = tree_verify_attn(q[:, order], parent2[None], K[:, :, rows], V[:, :, rows], [L])
    assert np.allclose(o2, o[:, order], rtol=1e-12, atol=1e-12), "tree relabel"


def read_cape_golden():
    lines = [ln.strip() for ln in open(os.path.join(GOLDEN, "cape_mask_example.txt"))
             if ln.strip() and not ln.startswith("#")]
    gamma = int(lines[0].split()[1])
    pos = [0] + [int(x) for x in lines[1].split()[1:]]
    keep = np.array([[c == "1" for c in row] for row in lines[2:]])
    return gamma, pos, keep


def check_cape_mask_golden(cape_mask, tree_allowed_mask):
    """The hand-worked CaPE mask example, from its equation and from the
    ancestor rule on the equivalent tree (proposal spine + expansion leaves)."""
    gamma, pos, keep = read_cape_golden()
    assert np.array_equal(cape_mask(gamma, pos), keep), "CaPE mask vs hand-worked example"
    parent = [-1] + [i - 1 for i in range(1, gamma + 1)] + [pos[i] - 1 for i in range(gamma + 1, len(pos))]
    allowed = tree_allowed_mask(parent, 0)
    assert allowed[:, 0].all(), "x_t must be visible to every tree token"
    assert np.array_equal(allowed[1:, 1:], keep), "ancestor mask vs hand-worked CaPE mask"


def check_cape_mask_random(cape_mask, tree_allowed_mask, cape_tree):
    """On random CaPE shapes (S(p) in {7,5,3,1}, Section 3.2) the CaPE mask
    equals the ancestor-or-self mask of the linearized tree."""
    g = _rng(10)
    for _ in range(50):
        gamma = int(g.integers(1, 7))
        sizes = [int(x) for x in g.choice([1, 3, 5, 7], size=gamma)]
        parent, pos = cape_tree(sizes)
        allowed = tree_allowed_mask(parent, 0)
        assert np.array_equal(allowed[1:, 1:], cape_mask(gamma, pos)), "CaPE mask != ancestor mask"


# ---------------------------------------------------------------- acceptance
def read_accept_golden():
    ex, cur = [], None
    for ln in open(os.path.join(GOLDEN, "accept_examples.txt")):
        ln = ln.strip()
        if not ln or ln.startswith("#"):
            continue
        key, *vals = ln.split()
        if key == "example":
            cur = {"name": vals[0]}
            ex.append(cur)
        else:
            cur[key] = [int(v) for v in vals]
    return ex


def logits_with_argmax(argmax, vocab, g):
    lg = g.standard_normal((len(argmax), vocab)).astype(np.float32)
    for i, a in enumerate(argmax):
        lg[i, a] = lg[i].max() + 1.0
    return lg


def check_accept_golden(tree_accept):
    g = _rng(11)
    for ex in read_accept_golden():
        n = len(ex["parent"])
        lg = logits_with_argmax(ex["argmax"], 16, g)[None]
        path, ln, bonus = tree_accept(np.array([ex["draft"]]), np.array([ex["parent"]]), lg)
        want = ex["path"] + [-1] * (n - len(ex["path"]))
        assert list(path[0]) == want, ex["name"]
        assert int(ln[0]) == ex["len"][0] and int(bonus[0]) == ex["bonus"][0], ex["name"]


def brute_force_accept(draft, parent, argmax):
    """Enumerate every root-to-node path and keep the longest fully matching
    one (ties: the path ending at the lowest node index)."""
    n = len(parent)
    best = (0, 0)
    for c in range(n):
        chain = [c]
        while chain[-1] != 0:
            chain.append(int(parent[chain[-1]]))
        chain.reverse()
        if all(int(draft[chain[k + 1]]) == int(argmax[chain[k]]) for k in range(len(chain) - 1)):
            if (len(chain) - 1, -c) > (best[0], -best[1]):
                best = (len(chain) - 1, c)
    d, c = best
    chain = [c]
    while chain[-1] != 0:
        chain.append(int(parent[chain[-1]]))
    return chain[::-1], d, int(argmax[c])


def random_small_tree(g, n):
    return np.array([-1] + [int(g.integers(i)) for i in range(1, n)])


def check_accept_brute_force(tree_accept):
    g = _rng(12)
    for trial in range(300):
        n = int(g.integers(1, 13))
        vocab = int(g.integers(2, 5))          # tiny vocab: many matches and ties
        parent = random_small_tree(g, n)
        draft = g.integers(vocab, size=n)
        lg = g.integers(-2, 3, size=(n, vocab)).astype(np.float32)   # integer logits: frequent ties
        argmax = [min(v for v in range(vocab) if lg[i, v] == lg[i].max()) for i in range(n)]
        chain, d, bonus = brute_force_accept(draft, parent, argmax)
        path, ln, bo = tree_accept(draft[None], parent[None], lg[None])
        assert list(path[0][:d + 1]) == chain and all(path[0][d + 1:] == -1), f"trial {trial}"
        assert int(ln[0]) == d and int(bo[0]) == bonus, f"trial {trial}"


def check_accept_chain_is_sd(tree_accept):
    """On a chain, acceptance is plain SD: the longest matching prefix of the
    proposal, then the target's token after it (Section 2)."""
    g = _rng(13)
    for _ in range(100):
        n = int(g.integers(1, 10))
        vocab = 3
        draft = g.integers(vocab, size=n)
        lg = g.standard_normal((n, vocab)).astype(np.float32)
        a = [int(np.argmax(lg[i])) for i in range(n)]
        k = 0
        while k + 1 < n and draft[k + 1] == a[k]:
            k += 1
        path, ln, bo = tree_accept(draft[None], np.arange(-1, n - 1)[None], lg[None])
        assert int(ln[0]) == k and int(bo[0]) == a[k] and list(path[0][:k + 1]) == list(range(k + 1))


def check_accept_greedy_equivalence(tree_accept):
    """With distinct sibling tokens the kept tokens plus the bonus are exactly
    what greedy decoding with the target emits while the tree can follow it."""
    g = _rng(14)
    for _ in range(200):
        n = int(g.integers(2, 16))
        vocab = 16                               # > n, so siblings can always be distinct
        parent = random_small_tree(g, n)
        draft = np.zeros(n, dtype=np.int64)
        for p in range(n):
            kids = [c for c in range(n) if parent[c] == p]
            if kids:
                draft[kids] = g.choice(vocab, size=len(kids), replace=False)
        lg = (g.standard_normal((n, vocab)) * 0.1).astype(np.float32)
        for p in range(n):                       # make the target follow the tree often
            kids = [c for c in range(n) if parent[c] == p]
            if kids and g.random() < 0.7:
                lg[p, draft[kids[int(g.integers(len(kids)))]]] = 5.0
        a = np.argmax(lg, axis=1)
        node, emitted = 0, []
        while True:
            nxt = [c for c in range(n) if parent[c] == node and draft[c] == a[node]]
            if not nxt:
                emitted.append(int(a[node]))
                break
            node = nxt[0]
            emitted.append(int(draft[node]))
        path, ln, bo = tree_accept(draft[None], parent[None], lg[None])
        got = [int(draft[c]) for c in path[0][1:int(ln[0]) + 1]] + [int(bo[0])]
        assert got == emitted


def check_argmax_ties(row_argmax):
    lg = np.array([[1.0, 3.0, 3.0, 2.0], [5.0, 5.0, 5.0, 5.0], [-1.0, -2.0, -1.0, -3.0],
                   [0.0, -0.0, 0.0, -1.0]], dtype=np.float32)
    assert list(row_argmax(lg)) == [1, 0, 0, 0]


# ----------------------------------------------------------- CaPE expansion
def read_cape_expand_golden():
    examples, sizes, cur, case = [], [], None, None
    for ln in open(os.path.join(GOLDEN, "cape_expand_examples.txt")):
        ln = ln.strip()
        if not ln or ln.startswith("#"):
            continue
        key, *vals = ln.split()
        if key == "example":
            cur = {"name": vals[0], "prob": [], "cases": []}
            examples.append(cur)
        elif key == "root":
            cur["root"] = int(vals[0])
        elif key == "prob":
            cur["prob"].append([float(v) for v in vals])
        elif key == "case":
            case = {"max_tokens": int(vals[0]), "fixed": None if vals[1] == "-" else int(vals[1])}
            cur["cases"].append(case)
        elif key == "size":
            bits = np.array([int(vals[0], 16)], dtype=np.uint32)
            sizes.append((float(bits.view(np.float32)[0]), int(vals[1])))
        else:
            case[key] = [int(v) for v in vals]
    return examples, sizes


def check_cape_expand_golden(cape_expand, expansion_size):
    """The hand-worked expansions (basic, caps, fixed size 4, tie + clamp) and
    S(p) at the binary32 neighbours of its thresholds."""
    examples, sizes = read_cape_expand_golden()
    for p, k in sizes:
        assert expansion_size(np.float32(p)) == k, f"S({p!r})"
    for ex in examples:
        probs = np.array([ex["prob"]], dtype=np.float32)
        gamma = probs.shape[1]
        for case in ex["cases"]:
            tok, par, nn, conf, ku = cape_expand(probs, np.array([ex["root"]]), case["max_tokens"],
                                                 case["fixed"])
            m = len(case["tokens"])
            tag = f"{ex['name']} cap {case['max_tokens']} fixed {case['fixed']}"
            assert int(nn[0]) == m, tag
            assert list(tok[0, :m]) == case["tokens"], tag
            assert list(par[0, :m]) == case["parent"], tag
            assert list(ku[0]) == case["k"], tag
            assert all(tok[0, m:] == -1) and all(par[0, m:] == 0), tag + " padding"
            assert np.array_equal(conf[0], probs[0].max(axis=-1)), tag + " conf"
            assert tok.shape[1] == 1 + case["max_tokens"], tag
            assert gamma <= case["max_tokens"]


def _outranks(p, a, b):
    """Token a ranks before token b in distribution p (ties: lower id)."""
    pa, pb = float(p[a]) + 0.0, float(p[b]) + 0.0
    return pa > pb or (pa == pb and a < b)


def check_cape_expand_brute_force(cape_expand, expansion_size):
    """Tiny vocabularies with many ties: x_{t+i} outranks every other token and
    X_i is the one subset of its size whose members all outrank every
    non-member, found by enumerating all subsets."""
    g = _rng(20)
    levels = np.array([0.0, 0.05, 0.1, 0.2, 0.35, 0.65, 0.9], dtype=np.float32)
    for trial in range(200):
        V = int(g.integers(2, 9))
        gamma = int(g.integers(1, 4))
        probs = levels[g.integers(len(levels), size=(1, gamma, V))]
        tok, par, nn, conf, ku = cape_expand(probs, np.array([0]), 63)
        node = gamma + 1
        for i in range(1, gamma + 1):
            p = probs[0, i - 1]
            x = int(tok[0, i])
            assert all(_outranks(p, x, u) for u in range(V) if u != x), f"trial {trial} x"
            k = int(ku[0, i - 1])
            assert k == min(expansion_size(p[x]), V - 1), f"trial {trial} K"
            X = [int(t) for t in tok[0, node:node + k]]
            assert all(int(q) == i - 1 for q in par[0, node:node + k]), f"trial {trial} parent"
            node += k
            others = [u for u in range(V) if u != x]
            winners = [set(T) for T in itertools.combinations(others, k)
                       if all(_outranks(p, a, b) for a in T for b in others if b not in T)]
            assert len(winners) == 1 and set(X) == winners[0], f"trial {trial} set"
            assert all(_outranks(p, X[r], X[r + 1]) for r in range(k - 1)), f"trial {trial} order"
        assert int(nn[0]) == node


def _planted_rows(g, sizes, V):
    """One distribution per position whose maximum is a value with a known
    S(p) from Section 3.2's table; the rest of the mass is spread below it."""
    p_of_size = {1: 0.9, 3: 0.7, 5: 0.5, 7: 0.2}
    rows = []
    for k in sizes:
        pmax = p_of_size[k]
        rest = g.random(V - 1) + 0.5
        rest *= (1.0 - pmax) / rest.sum()
        row = np.insert(rest, int(g.integers(V)), pmax)
        rows.append(row)
    return np.array([rows], dtype=np.float32)


def check_cape_expand_mask(cape_expand, cape_mask, tree_allowed_mask):
    """The tree built from CaPE's sets, under the ancestor-or-self rule, gives
    exactly the CaPE mask equation of Section 3.2 for the linearized proposal
    (pos() from the set sizes the planted confidences dictate)."""
    g = _rng(21)
    for _ in range(60):
        gamma = int(g.integers(1, 6))
        sizes = [int(k) for k in g.choice([1, 3, 5, 7], size=gamma)]
        probs = _planted_rows(g, sizes, 64)
        tok, par, nn, conf, ku = cape_expand(probs, np.array([5]), 63)
        assert list(ku[0]) == sizes
        n = int(nn[0])
        assert n == 1 + gamma + sum(sizes)
        pos = [0] + list(range(1, gamma + 1)) + [j for j, k in enumerate(sizes, start=1) for _ in range(k)]
        allowed = tree_allowed_mask(par[0, :n], 0)
        assert np.array_equal(allowed[1:, 1:], cape_mask(gamma, pos)), "CaPE tree mask"
        # siblings are distinct tokens, so greedy acceptance has one answer
        for p in range(n):
            kids = [int(tok[0, c]) for c in range(1, n) if par[0, c] == p]
            assert len(kids) == len(set(kids)), "duplicate siblings"


def check_cape_expand_cap(cape_expand):
    """Under a binding cap every dropped expansion token ranks after every kept
    one (probability, then position, then rank), each kept set is a prefix of
    its uncapped set, and the fixed size 0 gives the plain proposal chain."""
    g = _rng(22)
    for trial in range(100):
        gamma = int(g.integers(1, 6))
        V = int(g.integers(10, 60))
        probs = g.dirichlet(np.full(V, 0.3), size=(1, gamma)).astype(np.float32)
        probs[0, :, :3] = np.round(probs[0, :, :3], 1)           # some cross-position ties
        full = cape_expand(probs, np.array([1]), 63)
        cap = int(g.integers(gamma, gamma + int(full[4].sum()) + 1))
        part = cape_expand(probs, np.array([1]), cap)

        def entries(res):
            tok, par, nn, conf, ku = res
            out, node = [], gamma + 1
            for i in range(1, gamma + 1):
                for r in range(int(ku[0, i - 1])):
                    t = int(tok[0, node])
                    out.append((float(probs[0, i - 1, t]) + 0.0, i, r, t))
                    node += 1
            return out

        e_full, e_part = entries(full), entries(part)
        kept = set(e_part)
        assert kept <= set(e_full), f"trial {trial}"
        assert len(e_part) == min(len(e_full), cap - gamma), f"trial {trial}"
        for i in range(1, gamma + 1):
            mine = [e for e in e_full if e[1] == i]
            km = [e for e in e_part if e[1] == i]
            assert km == mine[:len(km)], f"trial {trial} prefix"
        for d in set(e_full) - kept:
            for k in kept:
                assert (k[0] > d[0]) or (k[0] == d[0] and (k[1], k[2]) < (d[1], d[2])), f"trial {trial} order"
        assert np.array_equal(full[0][0, :gamma + 1], part[0][0, :gamma + 1])
        chain = cape_expand(probs, np.array([1]), gamma, fixed_k=0)
        assert int(chain[2][0]) == gamma + 1 and list(chain[1][0]) == [-1] + list(range(gamma))


# --------------------------------------------------------- KV-cache update
def read_kv_golden():
    seqs, cur = [], None
    for ln in open(os.path.join(GOLDEN, "kv_compact_example.txt")):
        ln = ln.strip()
        if not ln or ln.startswith("#"):
            continue
        key, *vals = ln.split()
        if key == "seq":
            cur = {}
            seqs.append(cur)
        else:
            cur[key] = [int(v) for v in vals]
    return seqs


def check_kv_compact_golden(kv_compact):
    seqs = read_kv_golden()
    B, S = len(seqs), len(seqs[0]["rows"])
    K = np.array([[s["rows"]] for s in seqs], dtype=np.float32)[..., None]    # [B, 1, S, 1]
    V = -K
    n = max(len(s["path"]) for s in seqs)
    path = np.full((B, n), -1, dtype=np.int32)
    for b, s in enumerate(seqs):
        path[b, :len(s["path"])] = s["path"]
    K2, V2, nl = kv_compact(K, V, [s["kv_len"][0] for s in seqs], path, [s["len"][0] for s in seqs])
    for b, s in enumerate(seqs):
        assert list(K2[b, 0, :, 0].astype(int)) == s["want"], f"seq {b} K"
        assert list((-V2[b, 0, :, 0]).astype(int)) == s["want"], f"seq {b} V"
        assert int(nl[b]) == s["new_len"][0], f"seq {b} length"
    assert S == K2.shape[2]


def check_kv_compact_attention(kv_compact, tree_verify_attn, cross_attn):
    """The kept cache is exactly what the accepted node attended to during
    verification: plain attention of that node's query over the compacted
    cache reproduces its tree-attention output (up to fp64 rounding)."""
    g = _rng(23)
    for _ in range(20):
        B, H, D = 2, 2, 8
        n = int(g.integers(1, 10))
        L = [int(g.integers(0, 12)) for _ in range(B)]
        S = max(L) + n + 2
        K = g.standard_normal((B, H, S, D)).astype(np.float32)
        V = g.standard_normal((B, H, S, D)).astype(np.float32)
        parent = np.stack([random_small_tree(g, n) for _ in range(B)])
        q = g.standard_normal((B, n, H, D)).astype(np.float32)
        ref = tree_verify_attn(q, parent, K, V, L)
        path = np.full((B, n), -1, dtype=np.int32)
        length, node = [], []
        for b in range(B):
            c = int(g.integers(n))
            chain = [c]
            while chain[-1] != 0:
                chain.append(int(parent[b, chain[-1]]))
            chain = chain[::-1]
            path[b, :len(chain)] = chain
            length.append(len(chain) - 1)
            node.append(c)
        K2, V2, nl = kv_compact(K, V, L, path, length)
        qd = np.stack([q[b, node[b]] for b in range(B)])[:, None]
        got = cross_attn(qd, K2, V2, nl)
        for b in range(B):
            assert np.allclose(got[b, 0], ref[b, node[b]], rtol=1e-12, atol=1e-12), "kept cache"


def check_kv_compact_chain_identity(kv_compact):
    """Accepting a chain prefix (path[k] = k) moves nothing: the buffers are
    returned unchanged and only the length grows."""
    g = _rng(24)
    K = g.standard_normal((3, 2, 4, 20, 8)).astype(np.float32)     # [layers, B, H, S, D]
    V = g.standard_normal((3, 2, 4, 20, 8)).astype(np.float32)
    path = np.array([[0, 1, 2, -1, -1, -1], [0, 1, 2, 3, 4, 5]], dtype=np.int32)
    K2, V2, nl = kv_compact(K, V, [3, 10], path, [2, 5])
    assert np.array_equal(K2, K) and np.array_equal(V2, V)
    assert list(nl) == [6, 16]


# ------------------------------------------------- speculative sampling
def read_spec_sample_golden():
    ex, cur = [], None
    for ln in open(os.path.join(GOLDEN, "spec_sample_examples.txt")):
        ln = ln.strip()
        if not ln or ln.startswith("#"):
            continue
        key, *vals = ln.split()
        if key == "example":
            cur = {"name": vals[0], "pt": [], "q": []}
            ex.append(cur)
        elif key in ("pt", "q"):
            cur[key].append([float(v) for v in vals])
        elif key in ("gamma", "vocab"):
            cur[key] = int(vals[0])
        elif key in ("draft", "out"):
            cur[key] = [int(v) for v in vals]
        else:
            cur[key] = [float(v) for v in vals]
    return ex


def spec_golden_arrays(ex):
    """(draft [1, g], q [1, g, V] fp32, target logits [1, g+1, V] fp32, u [1, g+1] fp32)."""
    with np.errstate(divide="ignore"):
        lg = np.log(np.array(ex["pt"], dtype=np.float64))
    lg = np.where(np.isfinite(lg), lg, -1e4).astype(np.float32)
    return (np.array([ex["draft"]], dtype=np.int32), np.array([ex["q"]], dtype=np.float32), lg[None],
            np.array([ex["u"]], dtype=np.float32))


def check_spec_sample_golden(spec_sample_accept):
    for ex in read_spec_sample_golden():
        n, tok = spec_sample_accept(*spec_golden_arrays(ex))
        assert [int(n[0]), int(tok[0])] == ex["out"], ex["name"]


def _first_token_law(spec_sample_accept, q, logits, grid=2000):
    """Law of the first emitted token when x_1 ~ q and u, v are uniform, for
    gamma = 1, measured by running the rule over midpoint grids: the accept
    probability of each x over a u grid, the residual draw over a v grid."""
    V = len(q)
    mid = ((np.arange(grid) + 0.5) / grid).astype(np.float32)
    law = np.zeros(V)
    acc_rate = 0.0
    for x in range(V):
        if q[x] == 0:
            continue
        draft = np.full((grid, 1), x, dtype=np.int32)
        qs = np.broadcast_to(q, (grid, 1, V)).astype(np.float32)
        lg = np.broadcast_to(logits, (grid, 2, V)).astype(np.float32)
        u = np.stack([mid, np.zeros(grid, np.float32)], axis=1)
        n, _ = spec_sample_accept(draft, qs, lg, u)
        acc = float(np.mean(n == 1))
        u_rej = np.stack([np.full(grid, 0.99999994, np.float32), mid], axis=1)
        n2, tok = spec_sample_accept(draft, qs, lg, u_rej)
        if acc < 1.0:
            assert np.all(n2 == 0), "u close to 1 must reject a token the target likes less"
            resid = np.bincount(tok, minlength=V) / grid
        else:
            resid = np.zeros(V)
        law[x] += q[x] * acc
        law += q[x] * (1.0 - acc) * resid
        acc_rate += q[x] * acc
    return law, acc_rate


def check_spec_sample_is_target_sampling(spec_sample_accept):
    """The defining property of speculative sampling: with x_1 drawn from the
    draft, the first emitted token is distributed as the target's own sample,
    and a proposal is accepted with probability sum_x min(p_T(x), p_D(x))
    (Section 4.1, "Metrics")."""
    g = _rng(30)
    for trial in range(6):
        V = int(g.integers(3, 7))
        q = g.dirichlet(np.full(V, 0.7)).astype(np.float32)
        logits = (g.standard_normal((2, V)) * 1.5).astype(np.float32)
        law, acc_rate = _first_token_law(spec_sample_accept, q, logits)
        p = np.exp(logits[0].astype(np.float64) - logits[0].max())
        p /= p.sum()
        assert np.abs(law - p).max() < 5e-3, f"trial {trial}: law {law} vs target {p}"
        alpha = np.minimum(p, q.astype(np.float64)).sum()
        assert abs(acc_rate - alpha) < 5e-3, f"trial {trial}: acceptance {acc_rate} vs {alpha}"


def check_spec_sample_same_model_accepts(spec_sample_accept):
    """A draft equal to the target (up to fp32 rounding) is always accepted
    for u below 1 - 1e-6, and the extra token is then the inverse-CDF draw
    from the last target row."""
    g = _rng(31)
    B, gamma, V = 40, 5, 50
    logits = (g.standard_normal((B, gamma + 1, V)) * 2).astype(np.float32)
    z = logits.astype(np.float64)
    q = np.exp(z - z.max(-1, keepdims=True))
    q = (q / q.sum(-1, keepdims=True)).astype(np.float32)[:, :gamma]
    draft = np.stack([[int(g.choice(V, p=q[b, i] / q[b, i].sum())) for i in range(gamma)] for b in range(B)])
    u = (g.random((B, gamma + 1)) * 0.999).astype(np.float32)
    n, tok = spec_sample_accept(draft.astype(np.int32), q, logits, u)
    assert np.all(n == gamma)
    for b in range(B):
        p = np.exp(z[b, gamma] - z[b, gamma].max())
        c = np.cumsum(p / p.sum())
        assert int(tok[b]) == int(np.searchsorted(c, float(u[b, gamma]), side="right"))


# ------------------------------------------------ grouped-query attention
def check_gqa_is_repeated_kv(cross_attn, tree_verify_attn):
    """Grouped-query attention (the cached heads fewer than the query heads, as
    in Mistral-7B) is multi-head attention over cached heads repeated so that
    each run of H / H_kv consecutive query heads sees its own copy."""
    g = _rng(40)
    for H, H_kv in ((8, 2), (6, 3), (4, 1), (4, 4)):
        B, D, n = 2, 16, 5
        L = [9, 4]
        S = max(L) + n
        K = g.standard_normal((B, H_kv, S, D)).astype(np.float32)
        V = g.standard_normal((B, H_kv, S, D)).astype(np.float32)
        Kr, Vr = np.repeat(K, H // H_kv, axis=1), np.repeat(V, H // H_kv, axis=1)
        qd = g.standard_normal((B, 1, H, D)).astype(np.float32)
        assert np.allclose(cross_attn(qd, K, V, L), cross_attn(qd, Kr, Vr, L), rtol=1e-12, atol=1e-12), (H, H_kv)
        qt = g.standard_normal((B, n, H, D)).astype(np.float32)
        parent = np.stack([random_small_tree(g, n) for _ in range(B)])
        assert np.allclose(tree_verify_attn(qt, parent, K, V, L), tree_verify_attn(qt, parent, Kr, Vr, L),
                           rtol=1e-12, atol=1e-12), (H, H_kv)
        # and a query head reads exactly its group's cached head: changing another
        # group's cache leaves it alone
        if H_kv > 1:
            K2 = K.copy()
            K2[:, 1:] += g.standard_normal(K2[:, 1:].shape).astype(np.float32)
            o1, o2 = cross_attn(qd, K, V, L), cross_attn(qd, K2, V, L)
            grp = H // H_kv
            assert np.allclose(o1[:, :, :grp], o2[:, :, :grp]) and not np.allclose(o1[:, :, grp:], o2[:, :, grp:])


# --------------------------------------------- training-time block mask
def read_block_golden():
    lines = [ln.strip() for ln in open(os.path.join(GOLDEN, "block_mask_example.txt"))
             if ln.strip() and not ln.startswith("#")]
    T = int(lines[0].split()[1])
    L = int(lines[1].split()[1])
    keep = np.array([[c == "1" for c in row] for row in lines[2:]])
    return T, L, keep


def check_block_mask_golden(block_mask):
    T, L, keep = read_block_golden()
    assert keep.shape == (T, T)
    assert np.array_equal(block_mask(T, L), keep), "block mask vs hand-worked example"


def check_block_attn_is_delayed_cross(block_cross_attn, cross_attn):
    """Each position j's training-time output is the inference-time
    cross-attention of its query over the cache of the blocks before j's own
    block (kv_len = L * block(j)): the delayed cache the block mask simulates.
    Positions of the first block, and past a sequence's end, get zeros."""
    g = _rng(41)
    for H, H_kv, L in ((4, 4, 5), (4, 2, 3), (2, 1, 7)):
        B, T, D = 2, 23, 16
        seq_len = [23, 14]
        K = g.standard_normal((B, H_kv, T, D)).astype(np.float32)
        V = g.standard_normal((B, H_kv, T, D)).astype(np.float32)
        q = g.standard_normal((B, T, H, D)).astype(np.float32)
        out = block_cross_attn(q, K, V, seq_len, L)
        for b in range(B):
            for j in range(T):
                if j >= seq_len[b] or j < L:
                    assert np.all(out[b, j] == 0.0), (b, j)
                    continue
                kv = L * (j // L)
                want = cross_attn(q[b:b + 1, j:j + 1], K[b:b + 1], V[b:b + 1], [kv])
                assert np.allclose(out[b, j], want[0, 0], rtol=1e-12, atol=1e-12), (H, L, b, j)
