"""The library's calls captured into a CUDA graph and replayed give the same
bytes as eager calls (every kernel is deterministic; the cross-attention
merge is a programmatic dependent launch; the chunk-claim and arrival
counters are re-armed inside the kernels, so a replay starts clean)."""
import numpy as np
import pytest
import torch

from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build, synth

from gpu_util import dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    gb.lib()


def test_round_replays_bit_identical():
    w = synth.Workload("graph", B=3, H=8, D=128, dtype="bf16", kv_len=(900, 60, 2500), n=26, tree="random",
                       max_depth=5, max_branch=4, gamma=2, vocab=4000, logit_std=1.0, p_accept=0.7, seed=21)
    case = synth.make_case(w, garbage="zero")
    B, H, S_cap, D = case["K"].shape
    n = w.n
    K, V = dev(case["K"]), dev(case["V"])
    kv = dev(np.asarray(w.kv_len, np.int32))
    qd = [dev(case["q_draft"][i]) for i in range(w.gamma)]
    qt, par = dev(case["q_tree"]), dev(case["parent_idx"].astype(np.int32))
    draft, logits = dev(case["draft_tokens"].astype(np.int32)), dev(case["target_logits"])
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16)
    ws = torch.zeros(gb.glide_attn_workspace_bytes(desc, n), dtype=torch.uint8, device="cuda")
    wsa = torch.zeros(gb.glide_accept_workspace_bytes(B, n), dtype=torch.uint8, device="cuda")
    probs = dev(synth.draft_probs(22, B, 5, w.vocab))
    roots = dev(synth.root_tokens(22, B, w.vocab))
    wsc = torch.zeros(gb.glide_cape_workspace_bytes(B, 5, w.vocab), dtype=torch.uint8, device="cuda")
    sq = synth.draft_probs(23, B, 4, w.vocab)
    s_d, s_q = dev(synth.sample_tokens(23, sq)), dev(sq)
    s_l, s_u = dev(synth.target_logits_near(23, sq, 0.7)), dev(synth.uniforms(23, (B, 5)))
    wss = torch.zeros(gb.glide_sample_workspace_bytes(B, 4), dtype=torch.uint8, device="cuda")

    outs = {
        "cross": [torch.zeros(B, 1, H, D, device="cuda") for _ in range(w.gamma)],
        "tree": torch.zeros(B, n, H, D, device="cuda"),
        "path": torch.zeros(B, n, dtype=torch.int32, device="cuda"),
        "len": torch.zeros(B, dtype=torch.int32, device="cuda"),
        "bonus": torch.zeros(B, dtype=torch.int32, device="cuda"),
        "tok": torch.zeros(B, 33, dtype=torch.int32, device="cuda"),
        "tpar": torch.zeros(B, 33, dtype=torch.int32, device="cuda"),
        "nn": torch.zeros(B, dtype=torch.int32, device="cuda"),
        "sn": torch.zeros(B, dtype=torch.int32, device="cuda"),
        "st": torch.zeros(B, dtype=torch.int32, device="cuda"),
    }
    st = torch.cuda.Stream()

    def round_():
        for i in range(w.gamma):
            gb.glide_cross_attn(qd[i], K, V, kv, w.max_kv_len, outs["cross"][i], ws, stream=st)
        gb.tree_verify_attn(qt, par, K, V, kv, w.max_kv_len, outs["tree"], ws, stream=st)
        gb.tree_accept(draft, par, logits, outs["path"], outs["len"], outs["bonus"], wsa, stream=st)
        gb.cape_expand(probs, roots, 32, outs["tok"], outs["tpar"], outs["nn"], wsc, stream=st)
        gb.spec_sample_accept(s_d, s_q, s_l, s_u, outs["sn"], outs["st"], wss, stream=st)

    def snapshot():
        torch.cuda.synchronize()
        flat = []
        for v in outs.values():
            for t in (v if isinstance(v, list) else [v]):
                flat.append(t.clone().cpu())
                t.zero_()
        torch.cuda.synchronize()
        return flat

    torch.cuda.synchronize()           # the inputs were made on the default stream
    with torch.cuda.stream(st):
        round_()
    eager = snapshot()
    graph = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(graph, stream=st):
        round_()
    torch.cuda.synchronize()
    snapshot()                         # capture does not run the work; clear whatever is there
    for rep in range(2):
        graph.replay()
        got = snapshot()
        for a, b in zip(eager, got):
            assert torch.equal(a, b), f"replay {rep} differs from the eager round"
    assert int(ws[:256].abs().sum()) == 0 and int(wsa[:256].abs().sum()) == 0
