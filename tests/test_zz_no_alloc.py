"""glide_cross_attn_noalloc: the cross-attention entry point for callers that
cannot allocate device memory at call time (an engine plugin whose enqueue
path must not allocate, a serving loop that bans allocator calls on its
per-token path).  Its scratch is the library's own fixed array instead of a
caller workspace, so this checks, through the C ABI, that two calls in a row
give what glide_cross_attn gives with a caller workspace, and that shapes too
large for the fixed array are refused.

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
