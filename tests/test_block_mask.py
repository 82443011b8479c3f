"""The draft's training-time cross-attention under the block-wise mask through
the C ABI against the CPU oracle, within the attention tolerance of gpu_util;
positions with nothing to attend to must be exactly zero."""
import numpy as np
import pytest
import torch

import oracle
from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

from gpu_util import assert_attn_close, dev, sample_pairs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


@pytest.mark.parametrize("B,T,H,H_kv,D,L,seq_len,max_ctas", [
    (2, 130, 4, 4, 128, 5, [130, 77], 0),     # the paper's L = 5, a ragged second sequence
    (2, 64, 8, 2, 64, 5, [64, 5], 0),         # grouped heads; a sequence inside its first block
    (1, 300, 32, 8, 128, 3, [300], 0),        # Mistral-7B heads: 16 positions per query tile
    (3, 200, 4, 4, 128, 5, [200, 199, 0], 3),  # few CTAs: split slabs, merges; an empty sequence
    (3, 200, 4, 4, 128, 5, [200, 199, 0], 1000),
    (1, 100, 2, 1, 64, 1, [100], 0),          # L = 1: plain "earlier positions only"
    (1, 50, 2, 2, 128, 64, [50], 0),          # L > T: every position in the first block
    (2, 1024, 4, 2, 128, 5, [1024, 901], 0),  # eight position tiles: full and masked key tiles
    (1, 700, 4, 4, 64, 7, [700], 0),          # D = 64 (four K/V stages), an odd number of tiles
    (1, 130, 128, 1, 64, 5, [130], 0),        # 128 query heads on one cached head
    (64, 64, 2, 2, 128, 5, [64] * 63 + [17], 0),  # many sequences of one tile each
    (2, 640, 2, 2, 128, 5, [640, 640], 2),    # two CTAs walk all ten tile pairs
])
def test_block_cross_attn(B, T, H, H_kv, D, L, seq_len, max_ctas):
    S_cap = (T + 15) // 16 * 16
    K = synth.normal_values(1000 + T, 1, (B, H_kv, S_cap, D), "bf16")
    V = synth.normal_values(1000 + T, 2, (B, H_kv, S_cap, D), "bf16")
    q = synth.normal_values(1000 + T, 3, (B, T, H, D), "bf16")
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16, H_kv=H_kv)
    ws = torch.zeros(gb.glide_block_attn_workspace_bytes(desc, T), dtype=torch.uint8, device="cuda")
    out = torch.full((B, T, H, D), float("nan"), device="cuda")
    gb.glide_block_cross_attn(dev(q), dev(K), dev(V), dev(np.asarray(seq_len, np.int32)), L, out, ws,
                              max_ctas=max_ctas)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    want = oracle.block_cross_attn(q, K, V, seq_len, L)
    for b, n in enumerate(seq_len):
        dead = [j for j in range(T) if j < L or j >= n]
        assert np.all(got[b, dead] == 0.0), "positions that see no key must be zero"
    assert np.isfinite(got).all()
    live = [(b, h) for b in range(B) for h in range(H) if seq_len[b] > L]
    if live:
        assert_attn_close(got, want, live, f"block mask T{T} H{H}/{H_kv} L{L}")


def _random_block_case(seed):
    """A seeded random shape: sequences, positions, heads and their grouping,
    head dim, block length, ragged lengths (some zero) and a forced CTA count."""
    g = np.random.default_rng(seed)
    D = int(g.choice([64, 128]))
    H_kv = int(g.choice([1, 2, 4]))
    H = H_kv * int(g.choice([1, 2, 4]))
    B = int(g.integers(1, 4))
    T = int(g.integers(1, 700))
    L = int(g.choice([1, 2, 3, 5, 7, 16, 200]))
    seq_len = [int(g.integers(0, T + 1)) if g.random() < 0.5 else T for _ in range(B)]
    max_ctas = int(g.choice([0, 0, 1, 2, 3, 5]))
    return B, T, H, H_kv, D, L, seq_len, max_ctas


@pytest.mark.parametrize("seed", range(12))
def test_block_cross_attn_random_shapes(seed):
    """Random shapes against the oracle; every output written, the device
    status clean (a wait that ran out would show here)."""
    B, T, H, H_kv, D, L, seq_len, max_ctas = _random_block_case(4200 + seed)
    S_cap = (T + 15) // 16 * 16
    K = synth.normal_values(5000 + seed, 1, (B, H_kv, S_cap, D), "bf16")
    V = synth.normal_values(5000 + seed, 2, (B, H_kv, S_cap, D), "bf16")
    q = synth.normal_values(5000 + seed, 3, (B, T, H, D), "bf16")
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16, H_kv=H_kv)
    ws = torch.zeros(gb.glide_block_attn_workspace_bytes(desc, T), dtype=torch.uint8, device="cuda")
    out = torch.full((B, T, H, D), float("nan"), device="cuda")
    gb.glide_block_cross_attn(dev(q), dev(K), dev(V), dev(np.asarray(seq_len, np.int32)), L, out, ws,
                              max_ctas=max_ctas)
    torch.cuda.synchronize()
    assert gb.glide_read_device_status(ws) == gb.GLIDE_OK
    got = out.cpu().numpy()
    assert np.isfinite(got).all(), "every output element is written"
    want = oracle.block_cross_attn(q, K, V, seq_len, L)
    for b, n in enumerate(seq_len):
        dead = [j for j in range(T) if j < L or j >= n]
        assert np.all(got[b, dead] == 0.0)
    live = [(b, h) for b in range(B) for h in range(H) if seq_len[b] > L]
    if live:
        assert_attn_close(got, want, live, f"block mask random case {seed}")


def test_block_cross_attn_rising_scores():
    """Keys whose norm grows along the sequence push each key tile's maximum
    score far above the previous ones, so the lazy reference max moves and O
    is rescaled in tensor memory between tiles of a work item."""
    B, T, H, D, L = 1, 1024, 2, 128, 5
    S_cap = T
    ramp = (1.0 + np.arange(S_cap) / 40.0)[None, None, :, None]
    K = synth.f32_to_bf16_bits((synth.normal_values(91, 1, (B, H, S_cap, D), "f32") * ramp).astype(np.float32))
    V = synth.normal_values(91, 2, (B, H, S_cap, D), "bf16")
    q = synth.normal_values(91, 3, (B, T, H, D), "bf16")
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16)
    ws = torch.zeros(gb.glide_block_attn_workspace_bytes(desc, T), dtype=torch.uint8, device="cuda")
    out = torch.full((B, T, H, D), float("nan"), device="cuda")
    gb.glide_block_cross_attn(dev(q), dev(K), dev(V), dev(np.asarray([T], np.int32)), L, out, ws)
    torch.cuda.synchronize()
    want = oracle.block_cross_attn(q, K, V, [T], L)
    assert_attn_close(out.cpu().numpy(), want, [(0, 0), (0, 1)], "block mask, rising scores")


def test_block_cross_attn_matches_inference_cross_attn():
    """A position's training-time output equals glide_cross_attn of its query
    over the cache of the earlier blocks (kv_len = L * block(j)): the delayed
    cache the mask simulates, on the GPU."""
    B, T, H, D, L = 1, 120, 8, 128, 5
    S_cap = 128
    K = synth.normal_values(77, 1, (B, H, S_cap, D), "bf16")
    V = synth.normal_values(77, 2, (B, H, S_cap, D), "bf16")
    q = synth.normal_values(77, 3, (B, T, H, D), "bf16")
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16)
    ws = torch.zeros(gb.glide_block_attn_workspace_bytes(desc, T), dtype=torch.uint8, device="cuda")
    out = torch.zeros(B, T, H, D, device="cuda")
    Kd, Vd, qd = dev(K), dev(V), dev(q)
    gb.glide_block_cross_attn(qd, Kd, Vd, dev(np.asarray([T], np.int32)), L, out, ws)
    wsc = torch.zeros(gb.glide_attn_workspace_bytes(desc, 1), dtype=torch.uint8, device="cuda")
    for j in (5, 7, 49, 50, 119):
        kv = L * (j // L)
        oc = torch.zeros(B, 1, H, D, device="cuda")
        gb.glide_cross_attn(qd[:, j:j + 1].contiguous(), Kd, Vd, dev(np.asarray([kv], np.int32)), kv, oc, wsc)
        torch.cuda.synchronize()
        a, c = out[:, j].cpu().numpy(), oc[:, 0].cpu().numpy()
        assert np.allclose(a, c, atol=2e-3, rtol=1e-2), f"position {j}: {np.abs(a - c).max()}"


def test_two_draft_layers():
    """A two-layer draft (N_D = 2, the 33B setting) pairs draft layer m with
    target layer N_T - N_D + m: one step is two cross-attention calls on two
    layers' caches (layer 2's query comes from layer 1's output, so the calls
    are sequential).  With the layers stacked in one [N_T, B, H, S_cap, D]
    cache, the calls take views of its top two layers."""
    N_T, B, H, D, kv = 4, 2, 4, 128, [300, 41]
    S_cap = 320
    Kall = synth.normal_values(88, 1, (N_T, B, H, S_cap, D), "bf16")
    Vall = synth.normal_values(88, 2, (N_T, B, H, S_cap, D), "bf16")
    Kd, Vd = dev(Kall), dev(Vall)
    kvd = dev(np.asarray(kv, np.int32))
    ws = torch.zeros(gb.glide_attn_workspace_bytes(gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16), 1),
                     dtype=torch.uint8, device="cuda")
    for m in (1, 2):
        l = N_T - 2 + m                     # 1-based target layer of draft layer m
        q = synth.normal_values(88, 10 + m, (B, 1, H, D), "bf16")
        out = torch.zeros(B, 1, H, D, device="cuda")
        gb.glide_cross_attn(dev(q), Kd[l - 1], Vd[l - 1], kvd, max(kv), out, ws)
        torch.cuda.synchronize()
        want = oracle.cross_attn(q, Kall[l - 1], Vall[l - 1], kv)
        assert_attn_close(out.cpu().numpy(), want, None, f"draft layer {m} on target layer {l}")


def test_block_cross_attn_bench_shape_sampled():
    """The bench's training shape at full size (B = 4, T = 2048, 32 heads,
    D = 128, L = 5: 137 GFLOP), in the launch configuration the bench times,
    compared with the oracle on sampled (sequence, head) pairs."""
    B, T, H, D, L = 4, 2048, 32, 128, 5
    K = synth.normal_values(4242, 1, (B, H, T, D), "bf16")
    V = synth.normal_values(4242, 2, (B, H, T, D), "bf16")
    q = synth.normal_values(4242, 3, (B, T, H, D), "bf16")
    desc = gb.make_desc(B, H, D, T, gb.GLIDE_BF16)
    ws = torch.zeros(gb.glide_block_attn_workspace_bytes(desc, T), dtype=torch.uint8, device="cuda")
    out = torch.full((B, T, H, D), float("nan"), device="cuda")
    gb.glide_block_cross_attn(dev(q), dev(K), dev(V), dev(np.full(B, T, np.int32)), L, out, ws)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    assert np.isfinite(got).all()
    pairs = sample_pairs(B, H, 6, seed=7)
    want = oracle.block_cross_attn(q, K, V, [T] * B, L, pairs=pairs)
    assert np.all(got[:, :L] == 0.0)
    assert_attn_close(got, want, pairs, "block mask at the bench shape")
