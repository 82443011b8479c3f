"""Thin Python binding of libglide's C ABI (include/glide.h).

Argument marshalling only: shapes, dtypes and pointers of torch tensors are
turned into the C call; every step of the path runs in the library's CUDA
kernels.  The functions carry the C names.  A missing library is an error,
never a fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import build as _build

_LIB: Optional[ctypes.CDLL] = None

GLIDE_OK = 0
GLIDE_ERR_INVALID = 1
GLIDE_ERR_UNSUPPORTED = 2
GLIDE_ERR_CUDA = 3
GLIDE_ERR_DEVICE_TIMEOUT = 4

GLIDE_BF16 = 0
GLIDE_F32 = 1
GLIDE_FLAG_FORCE_FMA = 1
GLIDE_FLAG_TILE64 = 2


class GlideError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {glide_status_str(status)} (status {status})")
        self.status = status


class AttnDesc(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("H", ctypes.c_int32), ("D", ctypes.c_int32),
                ("S_cap", ctypes.c_int32), ("dtype", ctypes.c_int), ("scale", ctypes.c_float),
                ("flags", ctypes.c_uint32), ("max_ctas", ctypes.c_int32), ("H_kv", ctypes.c_int32)]


_P = ctypes.c_void_p
_SIG = {
    "glide_abi_version": (ctypes.c_int32, []),
    "glide_status_str": (ctypes.c_char_p, [ctypes.c_int]),
    "glide_attn_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(AttnDesc), ctypes.c_int32]),
    "glide_accept_workspace_bytes": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32]),
    "glide_cross_attn": (ctypes.c_int, [ctypes.POINTER(AttnDesc), _P, _P, _P, _P, ctypes.c_int32, _P, _P,
                                        ctypes.c_size_t, _P]),
    "tree_verify_attn": (ctypes.c_int, [ctypes.POINTER(AttnDesc), _P, ctypes.c_int32, _P, _P, _P, _P,
                                        ctypes.c_int32, _P, _P, ctypes.c_size_t, _P]),
    "tree_accept": (ctypes.c_int, [_P, _P, _P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _P, _P, _P, _P,
                                   ctypes.c_size_t, _P]),
    "glide_cross_attn_noalloc": (ctypes.c_int, [ctypes.POINTER(AttnDesc), _P, _P, _P, _P, ctypes.c_int32, _P, _P]),
    "glide_validate_tree": (ctypes.c_int, [_P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]),
    "glide_read_device_status": (ctypes.c_int, [_P, _P]),
    "glide_noalloc_read_device_status": (ctypes.c_int, [_P]),
    "glide_noalloc_scratch": (ctypes.c_int, [ctypes.POINTER(ctypes.c_void_p)]),
    "glide_selftest_wait_timeout": (ctypes.c_int, [_P, ctypes.c_uint32, _P]),
    "glide_cape_workspace_bytes": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]),
    "cape_expand": (ctypes.c_int, [_P, _P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                   ctypes.c_int32, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "glide_kv_compact": (ctypes.c_int, [ctypes.POINTER(AttnDesc), ctypes.c_int32, ctypes.c_int64, _P, _P, _P,
                                        ctypes.c_int32, _P, _P, _P, _P]),
    "glide_sample_workspace_bytes": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32]),
    "glide_block_attn_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(AttnDesc), ctypes.c_int32]),
    "glide_block_cross_attn": (ctypes.c_int, [ctypes.POINTER(AttnDesc), _P, ctypes.c_int32, ctypes.c_int32, _P, _P,
                                              _P, _P, _P, ctypes.c_size_t, _P]),
    "spec_sample_accept": (ctypes.c_int, [_P, _P, _P, _P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _P, _P,
                                          _P, ctypes.c_size_t, _P]),
}


def library_path() -> str:
    return _build.LIB


def lib() -> ctypes.CDLL:
    """The loaded libglide.so (raises if it has not been built)."""
    global _LIB
    if _LIB is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(f"libglide.so not found at {path}: build it first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(path)
        for name, (res, args) in _SIG.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


def glide_abi_version() -> int:
    return int(lib().glide_abi_version())


def glide_status_str(status: int) -> str:
    return lib().glide_status_str(int(status)).decode()


def _check(status: int, where: str):
    if status != GLIDE_OK:
        raise GlideError(status, where)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return GLIDE_BF16
    if t.dtype == torch.float32:
        return GLIDE_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def make_desc(B: int, H: int, D: int, S_cap: int, dtype: int, scale: float = 0.0, flags: int = 0,
              max_ctas: int = 0, H_kv: int = 0) -> AttnDesc:
    """H query heads; H_kv cached heads (0: H; fewer: grouped-query attention)."""
    return AttnDesc(B, H, D, S_cap, dtype, scale, flags, max_ctas, H_kv)


def glide_attn_workspace_bytes(desc: AttnDesc, n_queries: int) -> int:
    return int(lib().glide_attn_workspace_bytes(ctypes.byref(desc), n_queries))


def glide_accept_workspace_bytes(B: int, n: int) -> int:
    return int(lib().glide_accept_workspace_bytes(B, n))


def _cache_desc(q: torch.Tensor, K: torch.Tensor, V: torch.Tensor, scale, flags, max_ctas) -> AttnDesc:
    """Descriptor from queries [B, nq, H, D] and caches [B, H_kv, S_cap, D]."""
    if K.dim() != 4 or V.shape != K.shape or K.dtype != V.dtype or q.dtype != K.dtype or q.dim() != 4:
        raise ValueError("K/V must be [B, H_kv, S_cap, D] of the queries' dtype")
    for t in (q, K, V):
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
    B, H_kv, S_cap, D = K.shape
    H = q.shape[2]
    return make_desc(B, H, D, S_cap, _dtype_code(K), scale, flags, max_ctas, H_kv=H_kv if H_kv != H else 0)


def glide_cross_attn(q_draft: torch.Tensor, K_cache: torch.Tensor, V_cache: torch.Tensor, kv_len: torch.Tensor,
                     max_kv_len: int, out: torch.Tensor, workspace: torch.Tensor, scale: float = 0.0,
                     flags: int = 0, max_ctas: int = 0, stream=None) -> torch.Tensor:
    """out[B,1,H,D] fp32 <- GliDe cross-attention of q_draft[B,1,H,D] over K/V[B,H,S_cap,D]."""
    desc = _cache_desc(q_draft, K_cache, V_cache, scale, flags, max_ctas)
    if tuple(q_draft.shape) != (desc.B, 1, desc.H, desc.D) or tuple(out.shape) != (desc.B, 1, desc.H, desc.D):
        raise ValueError("q_draft/out must be [B, 1, H, D]")
    if out.dtype != torch.float32 or kv_len.dtype != torch.int32:
        raise TypeError("out must be fp32 and kv_len int32")
    st = lib().glide_cross_attn(ctypes.byref(desc), q_draft.data_ptr(), K_cache.data_ptr(), V_cache.data_ptr(),
                                kv_len.data_ptr(), int(max_kv_len), out.data_ptr(), workspace.data_ptr(),
                                workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "glide_cross_attn")
    return out


def glide_cross_attn_noalloc(q_draft: torch.Tensor, K_cache: torch.Tensor, V_cache: torch.Tensor,
                             kv_len: torch.Tensor, max_kv_len: int, out: torch.Tensor, scale: float = 0.0,
                             flags: int = 0, max_ctas: int = 0, stream=None) -> torch.Tensor:
    """glide_cross_attn without a workspace, for callers that cannot allocate
    device memory at call time; the library's fixed scratch array is used
    (see include/glide.h for its size limit and the no-overlap rule)."""
    desc = _cache_desc(q_draft, K_cache, V_cache, scale, flags, max_ctas)
    if tuple(q_draft.shape) != (desc.B, 1, desc.H, desc.D) or tuple(out.shape) != (desc.B, 1, desc.H, desc.D):
        raise ValueError("q_draft/out must be [B, 1, H, D]")
    if out.dtype != torch.float32 or kv_len.dtype != torch.int32:
        raise TypeError("out must be fp32 and kv_len int32")
    st = lib().glide_cross_attn_noalloc(ctypes.byref(desc), q_draft.data_ptr(), K_cache.data_ptr(),
                                        V_cache.data_ptr(), kv_len.data_ptr(), int(max_kv_len), out.data_ptr(),
                                        _stream(stream))
    _check(st, "glide_cross_attn_noalloc")
    return out


def tree_verify_attn(q_tree: torch.Tensor, parent_idx: torch.Tensor, K_cache: torch.Tensor, V_cache: torch.Tensor,
                     kv_len: torch.Tensor, max_kv_len: int, out: torch.Tensor, workspace: torch.Tensor,
                     scale: float = 0.0, flags: int = 0, max_ctas: int = 0, stream=None) -> torch.Tensor:
    """out[B,n,H,D] fp32 <- tree-masked verification attention of q_tree[B,n,H,D]."""
    desc = _cache_desc(q_tree, K_cache, V_cache, scale, flags, max_ctas)
    n = q_tree.shape[1]
    if tuple(q_tree.shape) != (desc.B, n, desc.H, desc.D) or tuple(out.shape) != (desc.B, n, desc.H, desc.D):
        raise ValueError("q_tree/out must be [B, n, H, D]")
    if tuple(parent_idx.shape) != (desc.B, n) or parent_idx.dtype != torch.int32 or kv_len.dtype != torch.int32:
        raise TypeError("parent_idx must be int32 [B, n] and kv_len int32 [B]")
    st = lib().tree_verify_attn(ctypes.byref(desc), q_tree.data_ptr(), n, parent_idx.data_ptr(),
                                K_cache.data_ptr(), V_cache.data_ptr(), kv_len.data_ptr(), int(max_kv_len),
                                out.data_ptr(), workspace.data_ptr(), workspace.numel() * workspace.element_size(),
                                _stream(stream))
    _check(st, "tree_verify_attn")
    return out


def tree_accept(draft_tokens: torch.Tensor, parent_idx: torch.Tensor, target_logits: torch.Tensor,
                path: torch.Tensor, length: torch.Tensor, bonus: torch.Tensor, workspace: torch.Tensor,
                stream=None):
    """(path[B,n], len[B], bonus[B]) int32 <- greedy tree acceptance."""
    B, n, V = target_logits.shape
    if target_logits.dtype != torch.float32 or not target_logits.is_contiguous():
        raise TypeError("target_logits must be contiguous fp32 [B, n, V]")
    for t, shp in ((draft_tokens, (B, n)), (parent_idx, (B, n)), (path, (B, n)), (length, (B,)), (bonus, (B,))):
        if t.dtype != torch.int32 or tuple(t.shape) != shp or not t.is_contiguous():
            raise TypeError("token, parent and output tensors must be contiguous int32")
    st = lib().tree_accept(draft_tokens.data_ptr(), parent_idx.data_ptr(), target_logits.data_ptr(), B, n, V,
                           path.data_ptr(), length.data_ptr(), bonus.data_ptr(), workspace.data_ptr(),
                           workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "tree_accept")
    return path, length, bonus


def glide_cape_workspace_bytes(B: int, gamma: int, V: int) -> int:
    return int(lib().glide_cape_workspace_bytes(B, gamma, V))


def cape_expand(probs: torch.Tensor, root_token: torch.Tensor, max_tokens: int, draft_tokens: torch.Tensor,
                parent_idx: torch.Tensor, n_nodes: torch.Tensor, workspace: torch.Tensor,
                conf: Optional[torch.Tensor] = None, fixed_k: int = -1, stream=None):
    """(draft_tokens, parent_idx [B, 1+max_tokens], n_nodes [B]) int32 (and conf [B, gamma] fp32)
    <- CaPE expansion of the draft distributions probs [B, gamma, V] fp32."""
    if probs.dim() != 3 or probs.dtype != torch.float32 or not probs.is_contiguous():
        raise TypeError("probs must be contiguous fp32 [B, gamma, V]")
    B, gamma, V = probs.shape
    n_out = 1 + int(max_tokens)
    for t, shp in ((root_token, (B,)), (draft_tokens, (B, n_out)), (parent_idx, (B, n_out)), (n_nodes, (B,))):
        if t.dtype != torch.int32 or tuple(t.shape) != shp or not t.is_contiguous():
            raise TypeError("root, token, parent and count tensors must be contiguous int32 of the stated shapes")
    if conf is not None and (conf.dtype != torch.float32 or tuple(conf.shape) != (B, gamma)
                             or not conf.is_contiguous()):
        raise TypeError("conf must be contiguous fp32 [B, gamma]")
    st = lib().cape_expand(probs.data_ptr(), root_token.data_ptr(), B, gamma, V, int(max_tokens), int(fixed_k),
                           draft_tokens.data_ptr(), parent_idx.data_ptr(), n_nodes.data_ptr(),
                           conf.data_ptr() if conf is not None else None, workspace.data_ptr(),
                           workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "cape_expand")
    return draft_tokens, parent_idx, n_nodes


def glide_kv_compact(K_cache: torch.Tensor, V_cache: torch.Tensor, kv_len: torch.Tensor, path: torch.Tensor,
                     length: torch.Tensor, new_kv_len: torch.Tensor, stream=None) -> torch.Tensor:
    """In-place cache update after acceptance.  K_cache/V_cache are one layer
    [B, H, S_cap, D] or a stack [layers, B, H, S_cap, D] (contiguous)."""
    if K_cache.shape != V_cache.shape or K_cache.dtype != V_cache.dtype:
        raise ValueError("K and V caches must match")
    if not (K_cache.is_contiguous() and V_cache.is_contiguous()):
        raise ValueError("caches must be contiguous")
    if K_cache.dim() == 4:
        layers, (B, H, S_cap, D) = 1, K_cache.shape
    elif K_cache.dim() == 5:
        layers, B, H, S_cap, D = K_cache.shape
    else:
        raise ValueError("caches must be [B, H, S_cap, D] or [layers, B, H, S_cap, D]")
    n = path.shape[-1]
    for t, shp in ((kv_len, (B,)), (path, (B, n)), (length, (B,)), (new_kv_len, (B,))):
        if t.dtype != torch.int32 or tuple(t.shape) != shp or not t.is_contiguous():
            raise TypeError("kv_len, path, len and new_kv_len must be contiguous int32 of the stated shapes")
    desc = make_desc(B, H, D, S_cap, _dtype_code(K_cache))
    st = lib().glide_kv_compact(ctypes.byref(desc), layers, B * H * S_cap * D, K_cache.data_ptr(),
                                V_cache.data_ptr(), kv_len.data_ptr(), n, path.data_ptr(), length.data_ptr(),
                                new_kv_len.data_ptr(), _stream(stream))
    _check(st, "glide_kv_compact")
    return new_kv_len


def glide_sample_workspace_bytes(B: int, gamma: int) -> int:
    return int(lib().glide_sample_workspace_bytes(B, gamma))


def spec_sample_accept(draft_tokens: torch.Tensor, draft_probs: torch.Tensor, target_logits: torch.Tensor,
                       uniforms: torch.Tensor, n_accepted: torch.Tensor, next_token: torch.Tensor,
                       workspace: torch.Tensor, stream=None):
    """(n_accepted [B], next_token [B]) int32 <- speculative-sampling acceptance of the
    chain draft_tokens [B, gamma] (draft_probs [B, gamma, V], target_logits [B, gamma+1, V],
    uniforms [B, gamma+1])."""
    B, gamma = draft_tokens.shape
    V = target_logits.shape[-1]
    for t, shp, dt in ((draft_tokens, (B, gamma), torch.int32), (draft_probs, (B, gamma, V), torch.float32),
                       (target_logits, (B, gamma + 1, V), torch.float32), (uniforms, (B, gamma + 1), torch.float32),
                       (n_accepted, (B,), torch.int32), (next_token, (B,), torch.int32)):
        if t.dtype != dt or tuple(t.shape) != shp or not t.is_contiguous():
            raise TypeError("spec_sample_accept: tensor of wrong dtype, shape or layout")
    st = lib().spec_sample_accept(draft_tokens.data_ptr(), draft_probs.data_ptr(), target_logits.data_ptr(),
                                  uniforms.data_ptr(), B, gamma, V, n_accepted.data_ptr(), next_token.data_ptr(),
                                  workspace.data_ptr(), workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "spec_sample_accept")
    return n_accepted, next_token


def glide_block_attn_workspace_bytes(desc: AttnDesc, T: int) -> int:
    return int(lib().glide_block_attn_workspace_bytes(ctypes.byref(desc), int(T)))


def glide_block_cross_attn(q: torch.Tensor, K_cache: torch.Tensor, V_cache: torch.Tensor, seq_len: torch.Tensor,
                           L: int, out: torch.Tensor, workspace: torch.Tensor, scale: float = 0.0, max_ctas: int = 0,
                           stream=None) -> torch.Tensor:
    """out[B,T,H,D] fp32 <- the draft's training-time cross-attention of q[B,T,H,D] over the
    target's K/V[B,H_kv,S_cap,D] under the block-wise mask with blocks of L positions."""
    desc = _cache_desc(q, K_cache, V_cache, scale, 0, max_ctas)
    T = q.shape[1]
    if tuple(out.shape) != tuple(q.shape) or out.dtype != torch.float32 or not out.is_contiguous():
        raise ValueError("out must be contiguous fp32 [B, T, H, D]")
    if seq_len.dtype != torch.int32 or tuple(seq_len.shape) != (desc.B,):
        raise TypeError("seq_len must be int32 [B]")
    st = lib().glide_block_cross_attn(ctypes.byref(desc), q.data_ptr(), T, int(L), K_cache.data_ptr(),
                                      V_cache.data_ptr(), seq_len.data_ptr(), out.data_ptr(), workspace.data_ptr(),
                                      workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "glide_block_cross_attn")
    return out


def glide_validate_tree(parent_idx_host, require_root0: bool = True) -> int:
    arr = torch.as_tensor(parent_idx_host, dtype=torch.int32).contiguous()
    if arr.dim() == 1:
        arr = arr[None]
    return int(lib().glide_validate_tree(arr.data_ptr(), arr.shape[0], arr.shape[1], int(bool(require_root0))))


def glide_read_device_status(workspace: torch.Tensor, stream=None) -> int:
    return int(lib().glide_read_device_status(workspace.data_ptr(), _stream(stream)))


def glide_selftest_wait_timeout(workspace: torch.Tensor, limit_us: int, stream=None) -> int:
    """Launch the bounded-wait self-test kernel (see include/glide.h); returns the launch status."""
    return int(lib().glide_selftest_wait_timeout(workspace.data_ptr(), int(limit_us), _stream(stream)))


def glide_noalloc_read_device_status(stream=None) -> int:
    """Status recorded in glide_cross_attn_noalloc's fixed array since it was last read (then cleared)."""
    return int(lib().glide_noalloc_read_device_status(_stream(stream)))


def glide_noalloc_scratch() -> int:
    """Device address of glide_cross_attn_noalloc's fixed array on the current device."""
    p = ctypes.c_void_p()
    _check(lib().glide_noalloc_scratch(ctypes.byref(p)), "glide_noalloc_scratch")
    return int(p.value)
