"""CUDA path vs. the CPU oracle, element by element, through the C ABI.

Attention: within the tolerance of gpu_util (elementwise 2e-2 + 1e-2|o| and
relative L2 <= 1e-2 per (b, h)).  Acceptance: bit-exact.  The five evaluation
workloads run at full size and every output is compared; the largest one's
oracle runs over all of its (b, h) slabs in spawned worker processes."""
import numpy as np
import pytest
import torch

import oracle
from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

from gpu_util import GpuCase, assert_attn_close, attn_errors, dev, oracle_every_slab, sample_pairs

pytestmark = pytest.mark.gpu

NAMES = [w.name for w in synth.workloads()]
LARGE = "vicuna33b-long-b4"
_WANT = {}  # oracle outputs per workload: (cross [gamma, B, 1, H, D], tree [B, n, H, D])


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


@pytest.fixture(scope="module", params=NAMES)
def wcase(request):
    """One evaluation workload resident on the GPU; pytest groups the tests by it."""
    torch.cuda.empty_cache()
    w = synth.workload(request.param)
    c = GpuCase(w, synth.make_case(w, garbage="nan"))
    yield c
    del c
    _WANT.pop(request.param, None)
    torch.cuda.empty_cache()


def want_for(c: GpuCase):
    """The oracle's outputs for every (b, h) of the workload, computed once."""
    if c.w.name not in _WANT:
        if c.w.name == LARGE:
            _WANT[c.w.name] = oracle_every_slab(c.case)
        else:
            cr = np.stack([oracle.cross_attn(c.case["q_draft"][s], c.case["K"], c.case["V"], c.case["kv_len"])
                           for s in range(c.w.gamma)])
            tr = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"],
                                         c.case["kv_len"])
            _WANT[c.w.name] = (cr, tr)
    return _WANT[c.w.name]


def test_cross_attn_workloads(wcase):
    c = wcase
    want = want_for(c)[0]
    for step in range(c.w.gamma):
        got = c.cross(step)
        assert_attn_close(got, want[step], None, f"{c.w.name} step {step}")
        assert np.isfinite(got).all()
    assert c.workspaces_clean()


@pytest.mark.parametrize("kernel", ["fma", "auto"])
def test_tree_verify_workloads(wcase, kernel):
    c = wcase
    got = c.tree(flags=gb.GLIDE_FLAG_FORCE_FMA if kernel == "fma" else 0)
    assert_attn_close(got, want_for(c)[1], None, f"{c.w.name} {kernel}")
    assert c.workspaces_clean()


def test_oracle_every_slab_matches_direct_oracle(wcase):
    """The pooled per-slab oracle agrees with the direct oracle call on a few
    slabs (the same arithmetic, so exactly)."""
    c = wcase
    if c.w.name != LARGE:
        pytest.skip("the pooled oracle serves the largest workload")
    pairs = sample_pairs(c.B, c.H, 3, seed=1)
    cr, tr = want_for(c)
    d = oracle.cross_attn(c.case["q_draft"][1], c.case["K"], c.case["V"], c.case["kv_len"], pairs=pairs)
    t = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"], c.case["kv_len"],
                                pairs=pairs)
    for b, h in pairs:
        assert np.array_equal(cr[1][b, :, h], d[b, :, h]) and np.array_equal(tr[b, :, h], t[b, :, h])


def test_tree_accept_workloads(wcase):
    c = wcase
    path, ln, bonus = c.accept()
    wp, wl, wb = oracle.tree_accept(c.case["draft_tokens"], c.case["parent_idx"], c.case["target_logits"])
    assert np.array_equal(path, wp) and np.array_equal(ln, wl) and np.array_equal(bonus, wb)
    assert c.workspaces_clean()
    assert gb.glide_read_device_status(c.ws_acc) == gb.GLIDE_OK
    assert gb.glide_read_device_status(c.ws) == gb.GLIDE_OK


# ------------------------------------------------------------------ edge cases
def small_case(B, H, D, dtype, kv_len, n, seed, tree="random", garbage="nan"):
    w = synth.Workload(f"edge-{seed}", B=B, H=H, D=D, dtype=dtype, kv_len=tuple(kv_len), n=n, tree=tree,
                       max_depth=6, max_branch=4, gamma=1, vocab=97, logit_std=1.0, p_accept=0.7, seed=seed)
    case = synth.make_case(w, garbage=garbage)
    return GpuCase(w, case)


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("bf16", 64), ("f32", 128), ("f32", 64)])
def test_cross_ragged_tails(dtype, D):
    kv = [1, 31, 32, 33, 63, 65, 129]
    c = small_case(len(kv), 3, D, dtype, kv, 4, seed=11 + D)
    for max_ctas in (0, 1, 2, 7, 1000):
        got = c.cross(max_ctas=max_ctas)
        want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], c.case["kv_len"])
        assert_attn_close(got, want, None, f"cross {dtype} D{D} ctas={max_ctas}")
    assert c.workspaces_clean()


def test_cross_empty_sequence_gives_zeros():
    c = small_case(3, 2, 128, "bf16", [40, 1, 7], 3, seed=21)
    kv = dev(np.array([40, 0, 7], dtype=np.int32))
    got = c.cross(kv_len=kv)
    assert np.array_equal(got[1], np.zeros_like(got[1]))
    want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], [40, 0, 7])
    assert_attn_close(got, want, [(0, 0), (0, 1), (2, 0), (2, 1)], "cross with an empty sequence")


@pytest.mark.parametrize("n", [1, 7, 33, 64])
@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64), ("bf16", 64)])
def test_tree_sizes(n, dtype, D):
    kv = [0, 5, 64, 100]
    c = small_case(len(kv), 2, D, dtype, kv, n, seed=31 + n + D)
    want = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"], kv)
    for flags in (gb.GLIDE_FLAG_FORCE_FMA, 0):
        for max_ctas in (0, 1, 3):
            got = c.tree(flags=flags, max_ctas=max_ctas)
            assert_attn_close(got, want, None, f"tree n={n} {dtype} D{D} flags={flags} ctas={max_ctas}")
    assert c.workspaces_clean()


def _random_attn_case(seed):
    """A seeded random shape: batch, heads, head dim, dtype, ragged cache
    lengths (some zero), tree size and shape, and a forced CTA count."""
    g = np.random.default_rng(seed)
    B = int(g.integers(1, 6))
    H = int(g.integers(1, 9))
    D = int(g.choice([64, 128]))
    dtype = str(g.choice(["bf16", "bf16", "f32"]))
    kv = [int(g.integers(0, 700)) if g.random() < 0.8 else 0 for _ in range(B)]
    if max(kv) == 0:
        kv[0] = 1
    n = int(g.choice([1, 2, 6, 17, 40, 64]))
    tree = str(g.choice(["random", "chain"]))
    max_ctas = int(g.choice([0, 0, 1, 3, 11, 1000]))
    return B, H, D, dtype, kv, n, tree, max_ctas


@pytest.mark.parametrize("seed", range(12))
def test_random_shapes(seed):
    """Cross-attention and tree verification of random shapes against the
    oracle, with the workspace left clean (no wait ran out, counters re-armed)."""
    B, H, D, dtype, kv, n, tree, max_ctas = _random_attn_case(6100 + seed)
    c = small_case(B, H, D, dtype, kv, n, seed=6100 + seed, tree=tree)
    live = [(b, h) for b in range(B) for h in range(H) if kv[b] > 0]
    got = c.cross(max_ctas=max_ctas)
    want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], kv)
    for b in range(B):
        if kv[b] == 0:
            assert np.array_equal(got[b], np.zeros_like(got[b]))
    if live:
        assert_attn_close(got, want, live, f"cross random case {seed}")
    want = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"], kv)
    for flags in (0, gb.GLIDE_FLAG_FORCE_FMA):
        assert_attn_close(c.tree(flags=flags, max_ctas=max_ctas), want, None,
                          f"tree random case {seed} flags={flags}")
    assert c.workspaces_clean()


def test_tree_chain_and_forest():
    c = small_case(2, 2, 128, "bf16", [70, 3], 9, seed=41, tree="chain")
    want = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"], [70, 3])
    assert_attn_close(c.tree(), want, None, "chain")
    forest = np.array([[-1, 0, -1, 2, 2, -1, 5, 6, 0]] * 2, dtype=np.int32)
    c.parent = dev(forest)
    want = oracle.tree_verify_attn(c.case["q_tree"], forest, c.case["K"], c.case["V"], [70, 3])
    for flags in (gb.GLIDE_FLAG_FORCE_FMA, 0):
        assert_attn_close(c.tree(flags=flags), want, None, "forest")


def test_peaked_softmax():
    """Queries scaled x4: attention far from uniform (score std 4)."""
    c = small_case(2, 3, 128, "bf16", [300, 77], 6, seed=51)
    q = c.case["q_tree"]
    qf = synth.bf16_bits_to_f32(q) * 4.0
    c.case["q_tree"] = synth.f32_to_bf16_bits(qf)
    c.q_tree = dev(c.case["q_tree"])
    want = oracle.tree_verify_attn(c.case["q_tree"], c.case["parent_idx"], c.case["K"], c.case["V"], [300, 77])
    for flags in (gb.GLIDE_FLAG_FORCE_FMA, 0):
        assert_attn_close(c.tree(flags=flags), want, None, "peaked tree")
    qd = synth.bf16_bits_to_f32(c.case["q_draft"][0]) * 4.0
    c.case["q_draft"] = synth.f32_to_bf16_bits(qd)[None]
    c.q_draft = [dev(c.case["q_draft"][0])]
    want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], [300, 77])
    assert_attn_close(c.cross(), want, None, "peaked cross")


def test_repeated_calls_reuse_workspace():
    c = small_case(3, 4, 128, "bf16", [500, 130, 9], 12, seed=61)
    a = [c.cross(max_ctas=5) for _ in range(3)]
    t = [c.tree(max_ctas=5) for _ in range(3)]
    acc = [c.accept() for _ in range(3)]
    assert all(np.array_equal(a[0], x) for x in a[1:])
    assert all(np.array_equal(t[0], x) for x in t[1:])
    assert all(all(np.array_equal(u, v) for u, v in zip(acc[0], x)) for x in acc[1:])
    assert c.workspaces_clean()
    assert gb.glide_read_device_status(c.ws) == gb.GLIDE_OK


def test_negative_control_is_rejected():
    """The comparison must fail for an all-zero output and for a shuffled V."""
    c = small_case(1, 8, 128, "bf16", [2048], 6, seed=71, tree="chain")
    want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], c.case["kv_len"])
    got = c.cross()
    ok, _, rel = attn_errors(np.zeros_like(got), want)
    assert not (ok and rel <= 1e-2)
    ok, _, rel = attn_errors(got[:, :, ::-1, :].copy(), want)
    assert not (ok and rel <= 1e-2)


# --------------------------------------------------------------- acceptance
def accept_case(B, n, V, seed, tree="random", p=0.7):
    g = np.random.default_rng(seed)
    parents = np.stack([synth.random_tree(seed + b, n, 8, 5) if tree == "random" else synth.chain_tree(n)
                        for b in range(B)])
    toks = np.stack([synth.draft_tokens(seed + 100 + b, parents[b], V) if V >= 8 else
                     g.integers(V, size=n).astype(np.int32) for b in range(B)])
    lg = np.stack([synth.planted_logits(seed + 200 + b, parents[b], toks[b], V, 1.0, p) if V >= 8 else
                   g.integers(-1, 2, size=(n, V)).astype(np.float32) for b in range(B)])
    return parents.astype(np.int32), toks.astype(np.int32), lg.astype(np.float32)


def run_accept(parents, toks, lg):
    B, n, V = lg.shape
    ws = torch.zeros(gb.glide_accept_workspace_bytes(B, n), dtype=torch.uint8, device="cuda")
    path = torch.full((B, n), -7, dtype=torch.int32, device="cuda")
    ln = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    bonus = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    gb.tree_accept(dev(toks), dev(parents), dev(lg), path, ln, bonus, ws)
    torch.cuda.synchronize()
    assert int(ws.count_nonzero()) == 0
    return path.cpu().numpy(), ln.cpu().numpy(), bonus.cpu().numpy()


@pytest.mark.parametrize("B,n,V,tree,p", [(1, 1, 50, "random", 0.7), (5, 64, 32000, "random", 0.9),
                                          (3, 13, 1001, "chain", 1.0), (64, 26, 257, "random", 0.6),
                                          (7, 9, 3, "random", 0.7), (2, 40, 9000, "chain", 0.5),
                                          (1024, 4, 8, "random", 0.7)])
def test_accept_shapes(B, n, V, tree, p):
    parents, toks, lg = accept_case(B, n, V, seed=B * 1000 + n, tree=tree, p=p)
    got = run_accept(parents, toks, lg)
    want = oracle.tree_accept(toks, parents, lg)
    for gv, wv in zip(got, want):
        assert np.array_equal(gv, wv)


def test_accept_ties_and_signed_zero():
    lg = np.zeros((1, 3, 12), dtype=np.float32)
    lg[0, 0, [3, 7]] = 2.0           # tie between 3 and 7 -> 3
    lg[0, 1, :] = -1.0
    lg[0, 1, 5] = -0.0               # -0 ties +0 at index 9 -> 5 is lower
    lg[0, 1, 9] = 0.0
    lg[0, 2, :] = -3.0
    parents = np.array([[-1, 0, 1]], dtype=np.int32)
    toks = np.array([[0, 3, 5]], dtype=np.int32)
    got = run_accept(parents, toks, lg)
    want = oracle.tree_accept(toks, parents, lg)
    assert list(got[0][0]) == list(want[0][0]) == [0, 1, 2] and got[1][0] == want[1][0] == 2
    assert got[2][0] == want[2][0] == 0


def test_accept_many_chunks_per_warp():
    """300 sequences of 64 nodes over 16384 logits: 76800 chunks of 4096
    logits on 152 CTAs of 14 consumer warps, so every warp counts more than a
    full batch of 32 chunks and some warps complete several sequences in one
    batch."""
    parents, toks, lg = accept_case(300, 64, 16384, seed=777, p=0.8)
    got = run_accept(parents, toks, lg)
    want = oracle.tree_accept(toks, parents, lg)
    for gv, wv in zip(got, want):
        assert np.array_equal(gv, wv)


def test_accept_ties_across_chunks_and_infinite_rows():
    """Equal maxima in different 4096-logit chunks of a row go to the lowest
    index, -0 equals +0 across chunks, a maximum in a row's ragged last chunk
    is found, and a row of -inf has its argmax at 0 (as numpy's)."""
    V = 32000
    lg = np.random.default_rng(5).standard_normal((2, 4, V)).astype(np.float32)
    lg[0, 0, [20000, 100, 31999]] = 9.0            # ties in chunks 4, 0 and 7 -> 100
    lg[0, 1, :] = -1.0
    lg[0, 1, [12288 + 5, 4096 * 7 + 3]] = 0.0      # +0 in chunk 3 ...
    lg[0, 1, 8191] = -0.0                           # ... -0 in chunk 1 wins by index
    lg[0, 2, 31999] = 50.0                          # the last logit of the ragged chunk
    lg[0, 3, :] = -np.inf
    lg[1] = lg[0, ::-1]
    parents = np.array([[-1, 0, 1, 2]] * 2, dtype=np.int32)
    a = oracle.row_argmax(lg)
    toks = np.stack([np.r_[0, a[b, :3]] for b in range(2)]).astype(np.int32)   # every edge matches
    got = run_accept(parents, toks, lg)
    want = oracle.tree_accept(toks, parents, lg)
    assert list(a[0]) == [100, 8191, 31999, 0]
    for gv, wv in zip(got, want):
        assert np.array_equal(gv, wv)
    assert list(got[1]) == [3, 3] and list(got[2]) == [0, 100]


def test_accept_invalid_parents_are_safe():
    """Parent arrays that break the contract (out of range, a second root,
    a parent after its child) give meaningless but well-formed results: no
    fault, a clean workspace, and a path that is a chain of matched edges
    from node 0 to a deepest node whose whole parent chain is valid and
    matched (the documented rule: a parent outside [0, c) makes node c
    unreachable)."""
    g = np.random.default_rng(31)
    B, n, V = 6, 64, 1000
    parents, toks, lg = accept_case(B, n, V, seed=4242, p=0.9)
    for b in range(B):
        for c in range(1, n):
            if g.random() < 0.12:
                parents[b, c] = int(g.choice([-1, -5, c, c + 3, n + 7, 2 ** 30]))
    path, ln, bonus = run_accept(parents, toks, lg)
    a = oracle.row_argmax(lg)
    for b in range(B):
        def chain(c):   # the root path of c, or None when it leaves [0, c) or an edge does not match
            out = [c]
            while c != 0:
                p = int(parents[b, c])
                if not (0 <= p < c) or toks[b, c] != a[b, p]:
                    return None
                out.append(p)
                c = p
            return out[::-1]
        ok = {c: chain(c) for c in range(n)}
        best = max((len(v) - 1, -c) for c, v in ok.items() if v is not None)
        node = -best[1]
        assert ln[b] == best[0] and bonus[b] == a[b, node]
        assert list(path[b, :ln[b] + 1]) == ok[node] and all(path[b, ln[b] + 1:] == -1)
