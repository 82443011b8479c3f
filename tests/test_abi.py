"""Host side of the C ABI (no GPU): the library builds and loads, exports every
entry point include/glide.h declares, and rejects bad arguments before any
CUDA call.  Only invalid arguments are passed here, so nothing is launched."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "glide.h")
FAKE = 0x10000  # 16-byte aligned, never dereferenced: every call below fails validation first


@pytest.fixture(scope="module")
def L():
    build.build()
    return gb.lib()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*[A-Za-z_][\w\s\*]*?\b([a-z_][a-z0-9_]*)\s*\(", src, flags=re.M)))


def test_exports_every_declared_symbol(L):
    names = declared_functions()
    assert len(names) >= 9, names
    for name in names:
        assert hasattr(L, name), f"libglide.so does not export {name}"


def test_noalloc_scratch_rejects_null(L):
    assert L.glide_noalloc_scratch(None) == gb.GLIDE_ERR_INVALID


def test_abi_version(L):
    assert gb.glide_abi_version() == 2


def test_status_strings(L):
    for s in range(5):
        assert gb.glide_status_str(s) and gb.glide_status_str(s) != "unknown status"
    assert gb.glide_status_str(99) == "unknown status"


def desc(**kw):
    d = dict(B=2, H=4, D=128, S_cap=300, dtype=gb.GLIDE_BF16, scale=0.0, flags=0, max_ctas=0)
    d.update(kw)
    return gb.make_desc(**d)


def test_workspace_sizes(L):
    d = desc()
    w1 = gb.glide_attn_workspace_bytes(d, 1)
    w64 = gb.glide_attn_workspace_bytes(d, 64)
    assert 0 < w1 < w64
    assert gb.glide_attn_workspace_bytes(d, 0) == 0
    assert gb.glide_attn_workspace_bytes(d, 65) == 0
    for bad in (dict(D=96), dict(B=0), dict(B=1025), dict(H=0), dict(S_cap=0), dict(dtype=7),
                dict(scale=-1.0), dict(scale=float("nan")), dict(scale=float("inf")), dict(max_ctas=-1)):
        assert gb.glide_attn_workspace_bytes(desc(**bad), 1) == 0, bad
    assert gb.glide_accept_workspace_bytes(4, 64) > 0
    assert gb.glide_accept_workspace_bytes(0, 4) == 0
    assert gb.glide_accept_workspace_bytes(4, 65) == 0


def cross(L, d, q=FAKE, K=FAKE, V=FAKE, kv=FAKE, max_kv=100, out=FAKE, ws=FAKE, wsb=1 << 40):
    return L.glide_cross_attn(ctypes.byref(d), q, K, V, kv, max_kv, out, ws, wsb, None)


def tree(L, d, n=5, q=FAKE, par=FAKE, K=FAKE, V=FAKE, kv=FAKE, max_kv=100, out=FAKE, ws=FAKE, wsb=1 << 40):
    return L.tree_verify_attn(ctypes.byref(d), q, n, par, K, V, kv, max_kv, out, ws, wsb, None)


def test_cross_rejects(L):
    d = desc()
    bad = [dict(q=None), dict(K=None), dict(V=None), dict(kv=None), dict(out=None), dict(ws=None),
           dict(max_kv=0), dict(max_kv=301), dict(wsb=16), dict(K=FAKE + 8), dict(out=FAKE + 4),
           dict(kv=FAKE + 2)]
    for b in bad:
        assert cross(L, d, **b) == gb.GLIDE_ERR_INVALID, b
    assert cross(L, desc(D=80)) == gb.GLIDE_ERR_INVALID
    assert L.glide_cross_attn(None, FAKE, FAKE, FAKE, FAKE, 10, FAKE, FAKE, 1 << 40, None) == gb.GLIDE_ERR_INVALID


def test_tree_rejects(L):
    d = desc()
    bad = [dict(n=0), dict(n=65), dict(par=None), dict(max_kv=296), dict(max_kv=-1), dict(wsb=100),
           dict(q=FAKE + 8), dict(par=FAKE + 1)]
    for b in bad:
        assert tree(L, d, **b) == gb.GLIDE_ERR_INVALID, b


def test_accept_rejects(L):
    def acc(draft=FAKE, par=FAKE, lg=FAKE, B=2, n=4, V=100, path=FAKE, ln=FAKE, bonus=FAKE, ws=FAKE, wsb=1 << 30):
        return L.tree_accept(draft, par, lg, B, n, V, path, ln, bonus, ws, wsb, None)
    for b in [dict(B=0), dict(n=0), dict(n=65), dict(V=0), dict(draft=None), dict(lg=None), dict(path=None),
              dict(ln=None), dict(bonus=None), dict(ws=None), dict(wsb=8), dict(lg=FAKE + 4),
              dict(path=FAKE + 2)]:
        assert acc(**b) == gb.GLIDE_ERR_INVALID, b


def test_cape_rejects(L):
    assert gb.glide_cape_workspace_bytes(4, 5, 32000) > 0
    for b in ((0, 5, 10), (4, 0, 10), (4, 64, 10), (4, 5, 0)):
        assert gb.glide_cape_workspace_bytes(*b) == 0, b

    def cape(probs=FAKE, root=FAKE, B=2, gamma=5, V=1000, max_tokens=32, fixed_k=-1, tok=FAKE, par=FAKE,
             nn=FAKE, conf=None, ws=FAKE, wsb=1 << 30):
        return L.cape_expand(probs, root, B, gamma, V, max_tokens, fixed_k, tok, par, nn, conf, ws, wsb, None)
    for b in [dict(B=0), dict(gamma=0), dict(V=0), dict(max_tokens=4), dict(max_tokens=64), dict(fixed_k=-2),
              dict(probs=None), dict(root=None), dict(tok=None), dict(par=None), dict(nn=None), dict(ws=None),
              dict(wsb=64), dict(probs=FAKE + 4), dict(ws=FAKE + 8), dict(tok=FAKE + 2), dict(conf=FAKE + 1)]:
        assert cape(**b) == gb.GLIDE_ERR_INVALID, b
    assert cape(fixed_k=8) == gb.GLIDE_ERR_UNSUPPORTED


def test_kv_compact_rejects(L):
    def comp(d=None, layers=1, stride=0, K=FAKE, V=FAKE, kv=FAKE, n=5, path=FAKE, ln=FAKE, new=FAKE + 256):
        d = d or desc()
        return L.glide_kv_compact(ctypes.byref(d), layers, stride, K, V, kv, n, path, ln, new, None)
    elems = 2 * 4 * 300 * 128
    for b in [dict(n=0), dict(n=65), dict(layers=0), dict(layers=2, stride=elems - 1), dict(layers=2, stride=elems + 4),
              dict(K=None), dict(V=None), dict(kv=None), dict(path=None), dict(ln=None), dict(new=None),
              dict(K=FAKE + 8), dict(path=FAKE + 2), dict(new=FAKE), dict(d=desc(D=80)), dict(d=desc(S_cap=4))]:
        assert comp(**b) == gb.GLIDE_ERR_INVALID, b


def test_validate_tree(L):
    assert gb.glide_validate_tree(np.array([-1, 0, 1, 1, 0])) == gb.GLIDE_OK
    assert gb.glide_validate_tree(np.array([[-1, 0, 0], [-1, 0, 1]])) == gb.GLIDE_OK
    assert gb.glide_validate_tree(np.array([-1, 0, 2])) == gb.GLIDE_ERR_INVALID      # parent not earlier
    assert gb.glide_validate_tree(np.array([-1, 0, -2])) == gb.GLIDE_ERR_INVALID     # below -1
    assert gb.glide_validate_tree(np.array([0, 0, 1])) == gb.GLIDE_ERR_INVALID       # node 0 not a root
    assert gb.glide_validate_tree(np.array([-1, 0, -1])) == gb.GLIDE_ERR_INVALID     # second root
    assert gb.glide_validate_tree(np.array([-1, 0, -1]), require_root0=False) == gb.GLIDE_OK  # forest


def test_binding_refuses_missing_library(monkeypatch, tmp_path):
    monkeypatch.setattr(gb, "_LIB", None)
    monkeypatch.setattr(gb, "library_path", lambda: str(tmp_path / "absent.so"))
    with pytest.raises(RuntimeError, match="not found"):
        gb.lib()


def test_spec_sample_rejects(L):
    assert gb.glide_sample_workspace_bytes(4, 5) > 0
    assert gb.glide_sample_workspace_bytes(0, 5) == 0 and gb.glide_sample_workspace_bytes(4, 0) == 0
    assert gb.glide_sample_workspace_bytes(4, 64) == 0

    def ss(d=FAKE, q=FAKE, lg=FAKE, u=FAKE, B=2, g=5, V=100, n=FAKE, t=FAKE, ws=FAKE, wsb=1 << 20):
        return L.spec_sample_accept(d, q, lg, u, B, g, V, n, t, ws, wsb, None)
    for b in [dict(B=0), dict(g=0), dict(g=64), dict(V=0), dict(d=None), dict(q=None), dict(lg=None), dict(u=None),
              dict(n=None), dict(t=None), dict(ws=None), dict(wsb=16), dict(lg=FAKE + 4), dict(q=FAKE + 2),
              dict(ws=FAKE + 8)]:
        assert ss(**b) == gb.GLIDE_ERR_INVALID, b


def test_grouped_query_descriptors(L):
    # H_kv must divide H and not exceed it
    for bad in (dict(H=8, H_kv=3), dict(H=4, H_kv=8), dict(H=4, H_kv=-1)):
        d = desc(**bad)
        assert gb.glide_attn_workspace_bytes(d, 1) == 0, bad
        assert cross(L, d) == gb.GLIDE_ERR_INVALID, bad
    # 32 query heads over 8 cached heads: 4 rows per node, so every tree of up to
    # 64 nodes fits the 256 query rows a cached head can serve
    d = desc(H=32, H_kv=8)
    assert gb.glide_attn_workspace_bytes(d, 64) > gb.glide_attn_workspace_bytes(d, 33) > 0
    # 64 query heads over 8: 8 rows per node, 32 nodes at most
    d = desc(H=64, H_kv=8)
    assert gb.glide_attn_workspace_bytes(d, 32) > 0 and gb.glide_attn_workspace_bytes(d, 33) == 0
    assert tree(L, d, n=33) == gb.GLIDE_ERR_UNSUPPORTED
    assert gb.glide_attn_workspace_bytes(desc(H=256, H_kv=1), 1) > 0       # 256 heads on one cache: 256 rows
    assert gb.glide_attn_workspace_bytes(desc(H=512, H_kv=1), 1) == 0      # 512 rows: beyond the limit
    assert cross(L, desc(H=512, H_kv=1)) == gb.GLIDE_ERR_UNSUPPORTED


def test_block_cross_attn_rejects(L):
    def blk(d=None, q=FAKE, T=100, Lb=5, K=FAKE, V=FAKE, sl=FAKE, out=FAKE, ws=FAKE, wsb=1 << 40):
        d = d or desc()
        return L.glide_block_cross_attn(ctypes.byref(d), q, T, Lb, K, V, sl, out, ws, wsb, None)
    assert gb.glide_block_attn_workspace_bytes(desc(), 100) > 0
    assert gb.glide_block_attn_workspace_bytes(desc(), 301) == 0
    for b in [dict(T=0), dict(T=301), dict(Lb=0), dict(q=None), dict(K=None), dict(sl=None), dict(out=None),
              dict(ws=None), dict(wsb=64), dict(q=FAKE + 8), dict(sl=FAKE + 2)]:
        assert blk(**b) == gb.GLIDE_ERR_INVALID, b
    assert blk(d=desc(dtype=gb.GLIDE_F32)) == gb.GLIDE_ERR_UNSUPPORTED
    # positions beyond 32-bit TMA row coordinates (B * T > 2^31), refused before any GPU call
    assert blk(d=desc(B=1024, H=1, S_cap=3_000_000), T=3_000_000) == gb.GLIDE_ERR_UNSUPPORTED
    assert gb.glide_block_attn_workspace_bytes(desc(B=1024, S_cap=4096), 4096) == 256  # the status word only
