"""Grouped-query attention (fewer cached heads than query heads, as in
Mistral-7B) through the C ABI against the CPU oracle: cross-attention and tree
verification on the tensor-core and CUDA-core paths, within the attention
tolerance of gpu_util."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

from gpu_util import assert_attn_close, dev

pytestmark = pytest.mark.gpu

T64 = gb.GLIDE_FLAG_TILE64


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


def make(B, H, H_kv, D, kv_len, n, dtype, seed, tree="random"):
    S_cap = (max(kv_len) + n + 15) // 16 * 16
    K = synth.normal_values(seed, 1, (B, H_kv, S_cap, D), dtype)
    V = synth.normal_values(seed, 2, (B, H_kv, S_cap, D), dtype)
    qd = synth.normal_values(seed, 3, (B, 1, H, D), dtype)
    qt = synth.normal_values(seed, 4, (B, n, H, D), dtype)
    if tree == "chain":
        parent = np.stack([synth.chain_tree(n) for _ in range(B)])
    else:
        parent = np.stack([synth.random_tree(seed + b, n, 6, 5) for b in range(B)])
    return K, V, qd, qt, parent.astype(np.int32)


def ws_for(B, H, H_kv, D, S_cap, n, dtype):
    d = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16 if dtype == "bf16" else gb.GLIDE_F32, H_kv=H_kv)
    return torch.zeros(gb.glide_attn_workspace_bytes(d, n), dtype=torch.uint8, device="cuda")


@pytest.mark.parametrize("B,H,H_kv,D,kv_len,dtype,flags,max_ctas", [
    (2, 32, 8, 128, [1000, 37], "bf16", 0, 0),      # Mistral-7B heads, tensor-core path
    (2, 32, 8, 128, [1000, 37], "bf16", gb.GLIDE_FLAG_FORCE_FMA, 0),
    (3, 8, 2, 64, [0, 513, 64], "bf16", 0, 0),      # an empty sequence gets zeros
    (3, 8, 2, 64, [0, 513, 64], "f32", 0, 0),       # CUDA-core path
    (1, 64, 1, 128, [2048], "bf16", 0, 0),          # one cached head for 64 query heads
    (1, 128, 1, 128, [2048], "bf16", 0, 0),         # 128 query rows: two row tiles
    (2, 256, 2, 64, [300, 0], "bf16", 0, 3),        # 128 rows per cached head, split shares, an empty sequence
    (1, 256, 1, 64, [500], "f32", 0, 0),            # 256 rows on the CUDA-core path
    (4, 32, 8, 128, [4096, 100, 2000, 16], "bf16", 0, 3),     # few CTAs: split (b, h), merged
    (4, 32, 8, 128, [4096, 100, 2000, 16], "bf16", 0, 1000),
    (2, 16, 4, 128, [300, 700], "f32", 0, 7),
    # the same cases on the 64-row kernel (GLIDE_FLAG_TILE64), and a group of 3,
    # which does not divide 128
    (2, 32, 8, 128, [1000, 37], "bf16", T64, 0),
    (3, 8, 2, 64, [0, 513, 64], "bf16", T64, 0),
    (4, 32, 8, 128, [4096, 100, 2000, 16], "bf16", T64, 3),
    (2, 24, 8, 128, [700, 50], "bf16", 0, 0),
])
def test_gqa_cross_attn(B, H, H_kv, D, kv_len, dtype, flags, max_ctas):
    K, V, qd, _, _ = make(B, H, H_kv, D, kv_len, 1, dtype, seed=700 + H + D)
    S_cap = K.shape[2]
    ws = ws_for(B, H, H_kv, D, S_cap, 1, dtype)
    out = torch.full((B, 1, H, D), float("nan"), device="cuda")
    gb.glide_cross_attn(dev(qd), dev(K), dev(V), dev(np.asarray(kv_len, np.int32)), max(max(kv_len), 1), out, ws,
                        flags=flags, max_ctas=max_ctas)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    want = oracle.cross_attn(qd, K, V, kv_len)
    for b, L in enumerate(kv_len):
        if L == 0:
            assert np.all(got[b] == 0.0), "an empty sequence must give zeros"
            want[b] = 0.0
    assert_attn_close(got, want, None, f"GQA cross H{H}/{H_kv} D{D} {dtype}")


@pytest.mark.parametrize("B,H,H_kv,D,kv_len,n,tree,dtype,flags,max_ctas", [
    (2, 32, 8, 128, [4096, 300], 6, "chain", "bf16", 0, 0),   # GliDe on Mistral-7B: gamma = 5 chain
    (2, 32, 8, 128, [4096, 300], 6, "chain", "bf16", T64, 0),
    (2, 32, 8, 128, [4096, 300], 6, "chain", "f32", 0, 0),
    (2, 8, 4, 128, [1500, 64], 26, "random", "bf16", 0, 0),   # 52 query rows per slab
    (1, 16, 4, 64, [777], 16, "random", "bf16", 0, 0),        # 64 rows: a full MMA
    (1, 16, 4, 64, [777], 16, "random", "bf16", gb.GLIDE_FLAG_FORCE_FMA, 0),
    (3, 32, 8, 128, [2000, 33, 900], 6, "random", "bf16", 0, 5),
    (3, 8, 4, 64, [0, 129, 64], 9, "random", "f32", 0, 1000),
    # CaPE-sized trees (33 nodes: 32 verified tokens plus the root) on
    # Mistral-7B's heads: 132 query rows per cached head, two row tiles of 128
    # (three of 64 with GLIDE_FLAG_TILE64)
    (2, 32, 8, 128, [3000, 200], 33, "random", "bf16", 0, 0),
    (2, 32, 8, 128, [3000, 200], 33, "random", "bf16", 0, 5),
    (2, 32, 8, 128, [3000, 200], 33, "random", "bf16", T64, 0),
    (2, 32, 8, 128, [3000, 200], 33, "random", "bf16", T64, 5),
    (2, 32, 8, 128, [3000, 200], 33, "random", "bf16", gb.GLIDE_FLAG_FORCE_FMA, 0),
    (3, 32, 8, 128, [0, 100, 1000], 33, "random", "bf16", 0, 0),   # no prefix; tree keys across a tile edge
    (3, 32, 8, 128, [0, 100, 1000], 33, "random", "bf16", 0, 7),
    (2, 32, 8, 128, [257, 2048], 33, "chain", "bf16", 0, 3),
    (1, 32, 8, 128, [1500], 64, "random", "bf16", 0, 0),       # 256 rows: the limit
    (1, 32, 8, 128, [1500], 64, "random", "bf16", 0, 1000),
    (1, 32, 8, 128, [1500], 64, "random", "bf16", T64, 1000),
    (2, 16, 8, 128, [900, 40], 40, "random", "bf16", 0, 0),    # group 2: 80 rows, one row tile of 128
    (2, 64, 8, 128, [600, 1300], 20, "random", "bf16", 0, 9),  # group 8: 160 rows
    (1, 32, 2, 128, [1100], 10, "random", "bf16", 0, 0),       # group 16: 160 rows
    (2, 24, 8, 128, [800, 300], 30, "random", "bf16", 0, 4),   # group 3 does not divide 128: 64-row tiles
    (2, 16, 4, 64, [700, 65], 20, "random", "bf16", 0, 7),     # 80 rows, D = 64
    (2, 16, 4, 64, [700, 65], 20, "random", "bf16", T64, 7),
    (2, 16, 4, 64, [700, 0], 20, "random", "f32", 0, 3),
])
def test_gqa_tree_verify(B, H, H_kv, D, kv_len, n, tree, dtype, flags, max_ctas):
    K, V, _, qt, parent = make(B, H, H_kv, D, kv_len, n, dtype, seed=800 + n + H, tree=tree)
    S_cap = K.shape[2]
    ws = ws_for(B, H, H_kv, D, S_cap, n, dtype)
    out = torch.full((B, n, H, D), float("nan"), device="cuda")
    gb.tree_verify_attn(dev(qt), dev(parent), dev(K), dev(V), dev(np.asarray(kv_len, np.int32)), max(kv_len),
                        out, ws, flags=flags, max_ctas=max_ctas)
    torch.cuda.synchronize()
    want = oracle.tree_verify_attn(qt, parent, K, V, kv_len)
    assert_attn_close(out.cpu().numpy(), want, None, f"GQA tree H{H}/{H_kv} n{n} {dtype}")


def test_gqa_equal_heads_is_multi_head():
    """H_kv = H through the descriptor is plain multi-head attention: the same
    output as a descriptor that leaves H_kv at 0."""
    B, H, D, kv_len, n = 2, 8, 128, [600, 90], 5
    K, V, qd, qt, parent = make(B, H, H, D, kv_len, n, "bf16", seed=900)
    S_cap = K.shape[2]
    Kd, Vd, kd, pd, q = dev(K), dev(V), dev(np.asarray(kv_len, np.int32)), dev(parent), dev(qt)
    outs = []
    L = gb.lib()
    for H_kv in (0, H):
        d = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16, H_kv=H_kv)
        ws = torch.zeros(gb.glide_attn_workspace_bytes(d, n), dtype=torch.uint8, device="cuda")
        out = torch.zeros(B, n, H, D, device="cuda")
        st = L.tree_verify_attn(ctypes.byref(d), q.data_ptr(), n, pd.data_ptr(), Kd.data_ptr(),
                                Vd.data_ptr(), kd.data_ptr(), max(kv_len), out.data_ptr(), ws.data_ptr(),
                                ws.numel(), None)
        assert st == gb.GLIDE_OK
        torch.cuda.synchronize()
        outs.append(out.cpu().numpy())
    assert np.array_equal(outs[0], outs[1])


def test_gqa_bench_shape_every_output():
    """Grouped-query attention on the bench's Mistral-7B shape at full size
    (B = 4, 32 query heads over 8 cached heads, D = 128, kv_len 16384, the
    6-node chain of GliDe with gamma = 5), both calls in the bench's launch
    configuration, every output compared with the oracle.  Each call runs
    three times on both tensor-core kernels: a race in the pipeline (the
    values arriving late from DRAM) shows as a changed result in some run."""
    B, H, H_kv, D, L, n = 4, 32, 8, 128, 16384, 6
    K, V, qd, qt, parent = make(B, H, H_kv, D, [L] * B, n, "bf16", seed=4343, tree="chain")
    S_cap = K.shape[2]
    ws = ws_for(B, H, H_kv, D, S_cap, n, "bf16")
    Kd, Vd, kv = dev(K), dev(V), dev(np.full(B, L, np.int32))
    want_c = oracle.cross_attn(qd, K, V, [L] * B)
    want_t = oracle.tree_verify_attn(qt, parent, K, V, [L] * B)
    qdd, qtd, pd = dev(qd), dev(qt), dev(parent)
    for flags in (0, T64):
        for rep in range(3):
            oc = torch.full((B, 1, H, D), float("nan"), device="cuda")
            ot = torch.full((B, n, H, D), float("nan"), device="cuda")
            gb.glide_cross_attn(qdd, Kd, Vd, kv, L, oc, ws, flags=flags)
            gb.tree_verify_attn(qtd, pd, Kd, Vd, kv, L, ot, ws, flags=flags)
            torch.cuda.synchronize()
            assert_attn_close(oc.cpu().numpy(), want_c, None, f"GQA cross-attention, bench shape, flags {flags}, run {rep}")
            assert_attn_close(ot.cpu().numpy(), want_t, None, f"GQA verification, bench shape, flags {flags}, run {rep}")


def test_gqa_cape_tree_bench_shape_every_output():
    """Verification of a 33-node CaPE tree on the bench's Mistral-7B shape at
    full size (B = 4, 32 query over 8 cached heads, D = 128, kv_len 16384:
    132 query rows per cached head, two row tiles of 128), in the bench's
    launch configuration, every output compared with the oracle, three runs."""
    B, H, H_kv, D, L, n = 4, 32, 8, 128, 16384, 33
    K, V, _, qt, parent = make(B, H, H_kv, D, [L] * B, n, "bf16", seed=4545)
    S_cap = K.shape[2]
    ws = ws_for(B, H, H_kv, D, S_cap, n, "bf16")
    want = oracle.tree_verify_attn(qt, parent, K, V, [L] * B)
    args = (dev(qt), dev(parent), dev(K), dev(V), dev(np.full(B, L, np.int32)), L)
    for rep in range(3):
        ot = torch.full((B, n, H, D), float("nan"), device="cuda")
        gb.tree_verify_attn(*args, ot, ws)
        torch.cuda.synchronize()
        assert_attn_close(ot.cpu().numpy(), want, None, f"GQA 33-node verification at the bench shape, run {rep}")


def test_gqa_many_sequences_on_128_row_tiles():
    """Three hundred sequences of short, ragged contexts (some empty) on the
    128-row kernel: a partition over 600 slabs, a batch table large enough
    that the launch takes fewer value stages, two row tiles per slab for the
    33-node trees, and the prefix-only mode with its zero rows, all against
    the oracle."""
    B, H, H_kv, D, n = 300, 8, 2, 128, 33
    kv_len = [int(x) for x in np.random.default_rng(5).integers(0, 260, B)]
    kv_len[0] = 0
    kv_len[7] = 0
    K, V, qd, qt, parent = make(B, H, H_kv, D, kv_len, n, "bf16", seed=951)
    S_cap = K.shape[2]
    ws = ws_for(B, H, H_kv, D, S_cap, n, "bf16")
    Kd, Vd, kv = dev(K), dev(V), dev(np.asarray(kv_len, np.int32))
    oc = torch.full((B, 1, H, D), float("nan"), device="cuda")
    ot = torch.full((B, n, H, D), float("nan"), device="cuda")
    gb.glide_cross_attn(dev(qd), Kd, Vd, kv, max(kv_len), oc, ws)
    gb.tree_verify_attn(dev(qt), dev(parent), Kd, Vd, kv, max(kv_len), ot, ws)
    torch.cuda.synchronize()
    want_c = oracle.cross_attn(qd, K, V, kv_len)
    for b, L in enumerate(kv_len):
        if L == 0:
            assert np.all(oc[b].cpu().numpy() == 0.0), "an empty sequence must give zeros"
            want_c[b] = 0.0
    assert_attn_close(oc.cpu().numpy(), want_c, None, "GQA cross, 300 ragged sequences")
    assert_attn_close(ot.cpu().numpy(), oracle.tree_verify_attn(qt, parent, K, V, kv_len), None,
                      "GQA verification, 300 ragged sequences")
