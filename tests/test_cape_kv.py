"""CUDA path vs. the CPU oracle for CaPE proposal expansion and the cache
update after acceptance, through the C ABI.  Both are integer/byte work:
bit-exact (tokens, parents, node counts, confidences, every cache byte)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

import pins
from gpu_util import dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


# ----------------------------------------------------------- CaPE expansion
def run_cape(probs: np.ndarray, root: np.ndarray, max_tokens: int, fixed_k=None, with_conf=True, ws=None,
             repeat=1):
    B, gamma, V = probs.shape
    n_out = 1 + max_tokens
    p = dev(probs.astype(np.float32))
    r = dev(root.astype(np.int32))
    tok = torch.full((B, n_out), 12345, dtype=torch.int32, device="cuda")
    par = torch.full((B, n_out), 12345, dtype=torch.int32, device="cuda")
    nn = torch.zeros(B, dtype=torch.int32, device="cuda")
    conf = torch.full((B, gamma), float("nan"), device="cuda") if with_conf else None
    if ws is None:
        ws = torch.zeros(gb.glide_cape_workspace_bytes(B, gamma, V), dtype=torch.uint8, device="cuda")
    for _ in range(repeat):
        gb.cape_expand(p, r, max_tokens, tok, par, nn, ws, conf=conf, fixed_k=-1 if fixed_k is None else fixed_k)
    torch.cuda.synchronize()
    return (tok.cpu().numpy(), par.cpu().numpy(), nn.cpu().numpy(),
            conf.cpu().numpy() if with_conf else None, ws)


def assert_cape_equal(probs, root, max_tokens, fixed_k=None, what="", **kw):
    tok, par, nn, conf, ws = run_cape(probs, root, max_tokens, fixed_k, **kw)
    o_tok, o_par, o_nn, o_conf, _ = oracle.cape_expand(probs, root, max_tokens, fixed_k)
    assert np.array_equal(nn, o_nn), f"{what}: n_nodes {nn} vs {o_nn}"
    assert np.array_equal(tok, o_tok), f"{what}: tokens"
    assert np.array_equal(par, o_par), f"{what}: parents"
    if conf is not None:
        assert np.array_equal(conf.view(np.uint32), o_conf.view(np.uint32)), f"{what}: conf"
    return tok, par, nn


def test_cape_golden_examples():
    """The hand-worked expansions of the golden file, on the GPU."""
    examples, _ = pins.read_cape_expand_golden()
    for ex in examples:
        probs = np.array([ex["prob"]], dtype=np.float32)
        for case in ex["cases"]:
            tok, par, nn, conf, _ = run_cape(probs, np.array([ex["root"]]), case["max_tokens"], case["fixed"])
            m = len(case["tokens"])
            assert int(nn[0]) == m
            assert list(tok[0, :m]) == case["tokens"] and list(par[0, :m]) == case["parent"], ex["name"]
            assert all(tok[0, m:] == -1) and all(par[0, m:] == 0)


def test_cape_threshold_neighbours():
    """Confidences at the binary32 neighbours of 0.3, 0.6, 0.8 pick the set
    sizes of the golden file (exact comparison on the device)."""
    _, sizes = pins.read_cape_expand_golden()
    V = 64
    rows = []
    for p, _ in sizes:
        row = np.full(V, (1.0 - p) / (V - 1) * 0.5, dtype=np.float32)
        row[7] = np.float32(p)
        rows.append(row)
    probs = np.array([rows], dtype=np.float32)
    tok, par, nn, conf, _ = run_cape(probs, np.array([0]), 63)
    o = oracle.cape_expand(probs, np.array([0]), 63)
    assert np.array_equal(tok, o[0]) and np.array_equal(par, o[1])
    assert list(o[4][0]) == [k for _, k in sizes]


@pytest.mark.parametrize("B,gamma,V,max_tokens,fixed_k", [
    (4, 5, 32000, 32, None),      # Vicuna vocabulary, the paper's cap
    (8, 5, 32000, 63, None),      # no binding cap
    (8, 5, 32000, 32, 4),         # Section 4's fixed size 4 (26 nodes)
    (2, 10, 32000, 40, None),
    (64, 5, 32000, 32, None),
    (3, 5, 32001, 32, None),      # ragged vocabulary (scalar path), partial last chunk
    (2, 7, 4097, 63, None),
    (5, 3, 7, 20, None),          # vocabulary smaller than a set
    (2, 4, 1, 10, None),          # a single token: empty sets
    (1, 63, 100, 63, None),       # every slot a proposal token, no room for sets
    (1, 1, 32000, 1, None),
    (2, 5, 32000, 10, 0),         # fixed size 0: the plain proposal chain
    (3, 6, 50257, 32, 7),
])
def test_cape_shapes(B, gamma, V, max_tokens, fixed_k):
    probs = synth.draft_probs(100 + B * gamma + V, B, gamma, V)
    root = synth.root_tokens(7, B, max(V, 1))
    assert_cape_equal(probs, root, max_tokens, fixed_k, f"B{B} g{gamma} V{V} cap{max_tokens} k{fixed_k}")


@pytest.mark.parametrize("V,quantum", [(1000, 1e-3), (32000, 1e-4), (32000, 0.05)])
def test_cape_ties(V, quantum):
    """Quantized distributions: many exact ties (and zeros) in the maximum,
    in the sets and across positions under the cap."""
    probs = synth.draft_probs(55, 6, 8, V, quantum=quantum)
    root = synth.root_tokens(8, 6, V)
    for cap in (8, 20, 32, 63):
        assert_cape_equal(probs, root, cap, None, f"V{V} q{quantum} cap{cap}")


def test_cape_degenerate_rows():
    """All-zero rows (p = 0), signed zeros, a uniform row and an exact 1.0."""
    V = 300
    probs = np.zeros((1, 4, V), dtype=np.float32)
    probs[0, 1] = -0.0
    probs[0, 1, 5] = 0.0
    probs[0, 2] = 1.0 / V
    probs[0, 3, 299] = 1.0
    assert_cape_equal(probs, np.array([3]), 40, None, "degenerate")


def test_cape_no_conf_and_workspace_reuse():
    probs = synth.draft_probs(9, 4, 5, 32000)
    root = synth.root_tokens(9, 4, 32000)
    tok, par, nn, _, ws = run_cape(probs, root, 32, with_conf=False, repeat=3)
    o = oracle.cape_expand(probs, root, 32)
    assert np.array_equal(tok, o[0]) and np.array_equal(par, o[1]) and np.array_equal(nn, o[2])
    B = 4
    counters = ws[256:256 + 4 * B].view(torch.int32)      # per-sequence arrival counters
    assert int(counters.abs().sum()) == 0, "sequence counters not re-armed"
    assert int(ws[:256].abs().sum()) == 0


def test_cape_tree_feeds_verifier():
    """The emitted arrays are valid trees for tree_accept (node 0 the only
    root), and their ancestor mask is the CaPE mask."""
    probs = synth.draft_probs(12, 6, 5, 32000)
    root = synth.root_tokens(12, 6, 32000)
    tok, par, nn, _, _ = run_cape(probs, root, 32)
    assert gb.glide_validate_tree(par, require_root0=True) == gb.GLIDE_OK
    o = oracle.cape_expand(probs, root, 32)
    for b in range(6):
        gamma = 5
        pos = [0] + list(range(1, gamma + 1)) + [j for j, k in enumerate(o[4][b], start=1) for _ in range(k)]
        n = int(nn[b])
        assert np.array_equal(oracle.tree_allowed_mask(par[b, :n], 0)[1:, 1:], oracle.cape_mask(gamma, pos))


# --------------------------------------------------------- KV-cache update
def run_compact(K: np.ndarray, V: np.ndarray, kv_len, path, length):
    Kd, Vd = dev(K), dev(V)
    kv = dev(np.asarray(kv_len, dtype=np.int32))
    pd = dev(np.asarray(path, dtype=np.int32))
    ld = dev(np.asarray(length, dtype=np.int32))
    nl = torch.full((K.shape[-4],), -7, dtype=torch.int32, device="cuda")
    gb.glide_kv_compact(Kd, Vd, kv, pd, ld, nl)
    torch.cuda.synchronize()

    def back(t):
        a = t.cpu()
        return a.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else a.numpy()
    return back(Kd), back(Vd), nl.cpu().numpy()


def accepted_paths(g, parent: np.ndarray):
    """A random accepted root path per tree: (path [B, n] -1 padded, len [B])."""
    B, n = parent.shape
    path = np.full((B, n), -1, dtype=np.int32)
    length = np.zeros(B, dtype=np.int32)
    for b in range(B):
        c = int(g.integers(n))
        chain = [c]
        while chain[-1] != 0:
            chain.append(int(parent[b, chain[-1]]))
        chain = chain[::-1]
        path[b, :len(chain)] = chain
        length[b] = len(chain) - 1
    return path, length


def kv_arrays(seed, shape, dtype):
    return synth.normal_values(seed, 1, shape, dtype), synth.normal_values(seed, 2, shape, dtype)


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("bf16", 64), ("f32", 128), ("f32", 64)])
@pytest.mark.parametrize("layers", [1, 3])
def test_kv_compact_random_trees(dtype, D, layers):
    g = np.random.default_rng(40 + D + layers)
    B, H, n = 5, 6, 26
    S = 400
    shape = (layers, B, H, S, D) if layers > 1 else (B, H, S, D)
    K, V = kv_arrays(3 + D, shape, dtype)
    kv_len = [int(x) for x in g.integers(0, S - n + 1, size=B)]
    parent = np.stack([synth.random_tree(60 + b, n, 6, 4) for b in range(B)]).astype(np.int32)
    path, length = accepted_paths(g, parent)
    gK, gV, gl = run_compact(K, V, kv_len, path, length)
    oK, oV, ol = oracle.kv_compact(K, V, kv_len, path, length)
    assert np.array_equal(gl, ol)
    assert np.array_equal(gK, oK) and np.array_equal(gV, oV)


def test_kv_compact_long_moves():
    """Paths that move more rows than one read-then-write batch (8): a leaf at
    node 1 then a 62-deep chain, and a chain over the even nodes."""
    B, H, S, D, n = 2, 3, 200, 128, 64
    K, V = kv_arrays(77, (B, H, S, D), "bf16")
    path = np.full((B, n), -1, dtype=np.int32)
    path[0, :63] = [0] + list(range(2, 64))                 # node 1 a leaf; 2..63 a chain under 0
    path[1, :32] = list(range(0, 64, 2))                     # even nodes form the chain
    length = np.array([62, 31], dtype=np.int32)
    kv_len = [100, 37]
    gK, gV, gl = run_compact(K, V, kv_len, path, length)
    oK, oV, ol = oracle.kv_compact(K, V, kv_len, path, length)
    assert np.array_equal(gl, ol) and np.array_equal(gK, oK) and np.array_equal(gV, oV)


def test_kv_compact_nothing_moves():
    """Chain prefixes and len 0 leave every byte in place."""
    B, H, S, D, n = 3, 4, 64, 64, 8
    K, V = kv_arrays(5, (B, H, S, D), "f32")
    path = np.array([[0, 1, 2, 3, -1, -1, -1, -1], [0] + [-1] * 7, list(range(8))], dtype=np.int32)
    gK, gV, gl = run_compact(K, V, [10, 0, 56], path, [3, 0, 7])
    assert np.array_equal(gK, K) and np.array_equal(gV, V)
    assert list(gl) == [14, 1, 64]


def test_kv_compact_clamps_out_of_range_lengths():
    """kv_len beyond S_cap - n is clamped to S_cap - n (like the attention
    kernels); the result equals the oracle at the clamped length."""
    B, H, S, D, n = 2, 2, 50, 128, 6
    K, V = kv_arrays(6, (B, H, S, D), "bf16")
    path = np.array([[0, 2, 5, -1, -1, -1], [0, 3, -1, -1, -1, -1]], dtype=np.int32)
    gK, gV, gl = run_compact(K, V, [S + 9, -4], path, [2, 1])
    oK, oV, ol = oracle.kv_compact(K, V, [S - n, 0], path, [2, 1])
    assert np.array_equal(gK, oK) and np.array_equal(gV, oV) and np.array_equal(gl, ol)


# ------------------------------------------------------------ whole round
def test_round_expand_verify_accept_compact():
    """One speculative round on the GPU, each step compared with the oracle
    on the oracle's own inputs: CaPE expansion of the draft distributions,
    tree verification, greedy acceptance, and the cache update."""
    B, H, D, V_voc, gamma, max_tokens = 3, 4, 128, 1000, 5, 32
    n = 1 + max_tokens
    probs = synth.draft_probs(31, B, gamma, V_voc)
    root = synth.root_tokens(31, B, V_voc)
    o_tok, o_par, o_nn, _, _ = oracle.cape_expand(probs, root, max_tokens)
    g_tok, g_par, g_nn, _, _ = run_cape(probs, root, max_tokens)
    assert np.array_equal(g_tok, o_tok) and np.array_equal(g_par, o_par) and np.array_equal(g_nn, o_nn)

    kv_len = [300, 17, 811]
    S = max(kv_len) + n + 5
    K, Vv = kv_arrays(32, (B, H, S, D), "bf16")
    q = synth.normal_values(32, 3, (B, n, H, D), "bf16")
    logits = np.stack([synth.planted_logits(33 + b, o_par[b], o_tok[b], V_voc, 2.0, 0.8) for b in range(B)])

    # verification
    desc_ws = torch.zeros(gb.glide_attn_workspace_bytes(gb.make_desc(B, H, D, S, gb.GLIDE_BF16), n),
                          dtype=torch.uint8, device="cuda")
    out = torch.full((B, n, H, D), float("nan"), device="cuda")
    Kd, Vd = dev(K), dev(Vv)
    kvd = dev(np.asarray(kv_len, dtype=np.int32))
    pard = dev(o_par)
    gb.tree_verify_attn(dev(q), pard, Kd, Vd, kvd, max(kv_len), out, desc_ws)
    want = oracle.tree_verify_attn(q, o_par, K, Vv, kv_len)
    from gpu_util import assert_attn_close
    assert_attn_close(out.cpu().numpy(), want, None, "round verify")

    # acceptance
    path = torch.zeros((B, n), dtype=torch.int32, device="cuda")
    ln = torch.zeros(B, dtype=torch.int32, device="cuda")
    bonus = torch.zeros(B, dtype=torch.int32, device="cuda")
    ws_acc = torch.zeros(gb.glide_accept_workspace_bytes(B, n), dtype=torch.uint8, device="cuda")
    gb.tree_accept(dev(o_tok), pard, dev(logits.astype(np.float32)), path, ln, bonus, ws_acc)
    o_path, o_len, o_bonus = oracle.tree_accept(o_tok, o_par, logits)
    assert np.array_equal(path.cpu().numpy(), o_path) and np.array_equal(ln.cpu().numpy(), o_len)
    assert np.array_equal(bonus.cpu().numpy(), o_bonus)
    assert int(o_len.max()) >= 1, "planted logits should accept something"

    # cache update
    nl = torch.zeros(B, dtype=torch.int32, device="cuda")
    gb.glide_kv_compact(Kd, Vd, kvd, dev(o_path), dev(o_len), nl)
    torch.cuda.synchronize()
    oK, oV, ol = oracle.kv_compact(K, Vv, kv_len, o_path, o_len)
    assert np.array_equal(nl.cpu().numpy(), ol)
    assert np.array_equal(Kd.cpu().view(torch.int16).numpy().view(np.uint16), oK)
    assert np.array_equal(Vd.cpu().view(torch.int16).numpy().view(np.uint16), oV)
