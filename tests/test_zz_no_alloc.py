"""glide_cross_attn_noalloc: the cross-attention entry point for callers that
cannot allocate device memory at call time (an engine plugin whose enqueue
path must not allocate, a serving loop that bans allocator calls on its
per-token path).  Its scratch is the library's own fixed array instead of a
caller workspace, so this checks, through the C ABI, that two calls in a row
give what glide_cross_attn gives with a caller workspace (multi-head and
grouped-query caches), that the array's device status reads OK after each
call and reports a wait that ran out, and that shapes too large for the fixed
array are refused.

The file name sorts last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

from gpu_util import GpuCase, assert_attn_close, dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


def _case(B, H, D, kv, seed):
    w = synth.Workload(f"noalloc-{seed}", B=B, H=H, D=D, dtype="bf16", kv_len=tuple(kv), n=4, tree="chain",
                       max_depth=4, max_branch=1, gamma=2, vocab=64, logit_std=1.0, p_accept=0.7, seed=seed)
    return GpuCase(w, synth.make_case(w, garbage="nan"))


@pytest.mark.parametrize("B,H,D,kv", [(3, 8, 128, [700, 33, 2049]), (2, 5, 64, [1, 300])])
def test_noalloc_matches_workspace_entry_point(B, H, D, kv):
    c = _case(B, H, D, kv, seed=500 + D)
    for step in range(2):                   # two calls in a row, different queries
        ref = c.cross(step=step)            # glide_cross_attn with a caller workspace
        out = torch.full((B, 1, H, D), float("nan"), device="cuda")
        gb.glide_cross_attn_noalloc(c.q_draft[step], c.K, c.V, c.kv_len, c.max_kv_len, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert_attn_close(got, ref.astype(np.float64), None, f"noalloc vs workspace, call {step}")
        want = oracle.cross_attn(c.case["q_draft"][step], c.case["K"], c.case["V"], c.case["kv_len"])
        assert_attn_close(got, want, None, f"noalloc vs oracle, call {step}")
        assert gb.glide_noalloc_read_device_status() == gb.GLIDE_OK


def test_noalloc_grouped_query_matches_workspace_entry_point():
    """H_kv < H: the grouped-query kernels keep a different partial layout in
    the same fixed array."""
    B, H, H_kv, D, kv = 2, 8, 2, 128, [300, 1025]
    S_cap = (max(kv) + 15) // 16 * 16
    Kh = synth.normal_values(900, 1, (B, H_kv, S_cap, D), "bf16")
    Vh = synth.normal_values(900, 2, (B, H_kv, S_cap, D), "bf16")
    K, V = dev(Kh), dev(Vh)
    kv_len = dev(np.asarray(kv, np.int32))
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16, H_kv=H_kv)
    ws = torch.zeros(gb.glide_attn_workspace_bytes(desc, 1), dtype=torch.uint8, device="cuda")
    for step in range(2):                   # two calls in a row, different queries
        qh = synth.normal_values(901 + step, 3, (B, 1, H, D), "bf16")
        q = dev(qh)
        ref = torch.full((B, 1, H, D), float("nan"), device="cuda")
        gb.glide_cross_attn(q, K, V, kv_len, max(kv), ref, ws)
        out = torch.full((B, 1, H, D), float("nan"), device="cuda")
        gb.glide_cross_attn_noalloc(q, K, V, kv_len, max(kv), out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert_attn_close(got, ref.cpu().numpy().astype(np.float64), None, f"grouped noalloc vs workspace, {step}")
        want = oracle.cross_attn(qh, Kh, Vh, kv)
        assert_attn_close(got, want, None, f"grouped noalloc vs oracle, call {step}")
        assert gb.glide_noalloc_read_device_status() == gb.GLIDE_OK


def test_noalloc_status_reports_a_wait_that_ran_out():
    """The bounded-wait self-test aimed at the fixed array records a timeout in
    its status word (no fault, no hang); a no-alloc call does not clear it, the
    reader reports it once and clears it, and calls keep working."""
    addr = gb.glide_noalloc_scratch()
    assert addr != 0 and addr % 256 == 0
    assert gb.glide_noalloc_read_device_status() == gb.GLIDE_OK
    st = gb.lib().glide_selftest_wait_timeout(addr, 20000, gb._stream(None))    # 20 ms limit
    assert st == gb.GLIDE_OK
    c = _case(2, 4, 64, [100, 7], seed=555)
    out = torch.full((2, 1, 4, 64), float("nan"), device="cuda")
    gb.glide_cross_attn_noalloc(c.q_draft[0], c.K, c.V, c.kv_len, c.max_kv_len, out)
    assert gb.glide_noalloc_read_device_status() == gb.GLIDE_ERR_DEVICE_TIMEOUT
    assert gb.glide_noalloc_read_device_status() == gb.GLIDE_OK            # the read cleared it
    got = out.cpu().numpy()
    want = oracle.cross_attn(c.case["q_draft"][0], c.case["K"], c.case["V"], c.case["kv_len"])
    assert_attn_close(got, want, None, "noalloc call after a planted timeout")


def test_noalloc_refuses_oversized_shape():
    L = gb.lib()
    # B*H = 8000 at D = 128 needs more scratch than the fixed 32 MiB array holds
    desc = gb.make_desc(8, 1000, 128, 64, gb.GLIDE_BF16)
    assert gb.glide_attn_workspace_bytes(desc, 1) > 32 << 20
    fake = 0x10000
    st = L.glide_cross_attn_noalloc(ctypes.byref(desc), fake, fake, fake, fake, 16, fake, None)
    assert st == gb.GLIDE_ERR_UNSUPPORTED
    assert gb.glide_status_str(st) == "unsupported shape or type"
    bad = gb.make_desc(2, 4, 96, 64, gb.GLIDE_BF16)      # D = 96 is not a supported head size
    assert L.glide_cross_attn_noalloc(ctypes.byref(bad), fake, fake, fake, fake, 16, fake, None) == \
        gb.GLIDE_ERR_INVALID
