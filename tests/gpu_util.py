"""Helpers for the GPU parity tests: upload seeded inputs, call the C ABI
through the binding, and compare with the oracle under the stated tolerance."""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np
import torch

from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import synth

# Tolerance for attention outputs (bf16 inputs, fp32 accumulation): elementwise
# |gpu - oracle| <= ATOL + RTOL * |oracle|, and, because near-uniform softmax
# makes outputs tiny at long contexts (an all-zero output would pass the
# absolute bound), the relative L2 error of every (b, h) block <= REL_L2.
ATOL = 2e-2
RTOL = 1e-2
REL_L2 = 1e-2


def dev(arr: np.ndarray, device="cuda") -> torch.Tensor:
    if arr.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(np.ascontiguousarray(arr)).to(device)


def attn_errors(got: np.ndarray, want: np.ndarray, pairs=None):
    """(elementwise ok, max abs err, max rel-L2 over (b, h)) for [B, nq, H, D] arrays."""
    B, nq, H, D = want.shape
    if pairs is None:
        pairs = [(b, h) for b in range(B) for h in range(H)]
    ok = True
    max_abs = 0.0
    max_rel = 0.0
    for b, h in pairs:
        g = got[b, :, h, :].astype(np.float64)
        o = want[b, :, h, :]
        err = np.abs(g - o)
        ok &= bool(np.all(err <= ATOL + RTOL * np.abs(o)))
        max_abs = max(max_abs, float(err.max()))
        max_rel = max(max_rel, float(np.linalg.norm(g - o) / max(np.linalg.norm(o), 1e-300)))
    return ok, max_abs, max_rel


def assert_attn_close(got, want, pairs=None, what=""):
    assert np.all(np.isfinite(got if pairs is None else np.stack([got[b, :, h] for b, h in pairs]))), what
    ok, max_abs, max_rel = attn_errors(got, want, pairs)
    assert ok and max_rel <= REL_L2, f"{what}: max|err|={max_abs:.3e} max relL2={max_rel:.3e}"
    return max_abs, max_rel


class GpuCase:
    """One workload's inputs on the device, plus workspaces."""

    def __init__(self, w: synth.Workload, case: dict):
        self.w = w
        self.case = case
        self.K = dev(case["K"])
        self.V = dev(case["V"])
        self.q_draft = [dev(case["q_draft"][i]) for i in range(case["q_draft"].shape[0])]
        self.q_tree = dev(case["q_tree"])
        self.parent = dev(case["parent_idx"].astype(np.int32))
        self.kv_len = dev(np.asarray(case["kv_len"], dtype=np.int32))
        self.draft = dev(case["draft_tokens"].astype(np.int32))
        self.logits = dev(case["target_logits"].astype(np.float32))
        self.B, self.H, self.S_cap, self.D = case["K"].shape
        self.n = case["q_tree"].shape[1]
        self.max_kv_len = int(max(case["kv_len"]))
        d = gb.make_desc(self.B, self.H, self.D, self.S_cap, gb.GLIDE_BF16 if case["K"].dtype == np.uint16
                         else gb.GLIDE_F32)
        self.ws = torch.zeros(gb.glide_attn_workspace_bytes(d, max(self.n, 1)), dtype=torch.uint8, device="cuda")
        self.ws_acc = torch.zeros(gb.glide_accept_workspace_bytes(self.B, self.n), dtype=torch.uint8, device="cuda")

    def cross(self, step=0, max_ctas=0, kv_len=None, max_kv_len=None):
        out = torch.full((self.B, 1, self.H, self.D), float("nan"), device="cuda")
        gb.glide_cross_attn(self.q_draft[step], self.K, self.V, self.kv_len if kv_len is None else kv_len,
                            self.max_kv_len if max_kv_len is None else max_kv_len, out, self.ws,
                            max_ctas=max_ctas)
        torch.cuda.synchronize()
        return out.cpu().numpy()

    def tree(self, flags=0, max_ctas=0):
        out = torch.full((self.B, self.n, self.H, self.D), float("nan"), device="cuda")
        gb.tree_verify_attn(self.q_tree, self.parent, self.K, self.V, self.kv_len, self.max_kv_len, out, self.ws,
                            flags=flags, max_ctas=max_ctas)
        torch.cuda.synchronize()
        return out.cpu().numpy()

    def accept(self):
        path = torch.full((self.B, self.n), -7, dtype=torch.int32, device="cuda")
        ln = torch.full((self.B,), -7, dtype=torch.int32, device="cuda")
        bonus = torch.full((self.B,), -7, dtype=torch.int32, device="cuda")
        gb.tree_accept(self.draft, self.parent, self.logits, path, ln, bonus, self.ws_acc)
        torch.cuda.synchronize()
        return path.cpu().numpy(), ln.cpu().numpy(), bonus.cpu().numpy()

    def workspaces_clean(self):
        """Status word and arrival counters of the attention workspace, and the
        whole acceptance workspace, are back to zero (partial slots are scratch)."""
        counted = 256 + ((4 * self.B * self.H + 255) // 256) * 256
        return int(self.ws[:counted].count_nonzero()) == 0 and int(self.ws_acc.count_nonzero()) == 0


def sample_pairs(B, H, k, seed=0):
    g = np.random.default_rng(seed)
    pairs = {(0, 0), (B - 1, H - 1)}
    while len(pairs) < min(k, B * H):
        pairs.add((int(g.integers(B)), int(g.integers(H))))
    return sorted(pairs)


def _oracle_slab(args):
    """Oracle outputs of one (sequence, head) slab: the gamma cross-attention
    steps and the tree verification over that slab's keys and values."""
    import oracle
    q_draft, q_tree, parent, Kbh, Vbh, L = args
    cross = np.stack([oracle.cross_attn(q_draft[i][None, None, None, :], Kbh[None, None], Vbh[None, None], [L])[0, 0, 0]
                      for i in range(q_draft.shape[0])])
    tree = oracle.tree_verify_attn(q_tree[None, :, None, :], parent[None], Kbh[None, None], Vbh[None, None], [L])[0, :, 0]
    return cross, tree


def oracle_every_slab(case: dict, workers: int = 0):
    """The oracle over every (b, h) slab of a case, spread over spawned
    single-threaded worker processes (spawned, so the CUDA context of this
    process is never forked).  Returns (cross [gamma, B, 1, H, D],
    tree [B, n, H, D]) in fp64."""
    K = case["K"]
    B, H, _, D = K.shape
    n = case["q_tree"].shape[1]
    gamma = case["q_draft"].shape[0]
    kv = [int(x) for x in case["kv_len"]]
    args = [(case["q_draft"][:, b, 0, h, :], case["q_tree"][b, :, h, :], case["parent_idx"][b],
             np.ascontiguousarray(K[b, h, :kv[b] + n]), np.ascontiguousarray(case["V"][b, h, :kv[b] + n]), kv[b])
            for b in range(B) for h in range(H)]
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    with mp.get_context("spawn").Pool(workers or os.cpu_count() or 1) as pool:
        res = pool.map(_oracle_slab, args, chunksize=1)
    cross = np.zeros((gamma, B, 1, H, D))
    tree = np.zeros((B, n, H, D))
    for (b, h), (c, t) in zip([(b, h) for b in range(B) for h in range(H)], res):
        cross[:, b, 0, h, :] = c
        tree[b, :, h, :] = t
    return cross, tree
