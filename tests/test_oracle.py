"""The CPU oracle against its pins (no GPU).

Each pin is run on the real oracle and must pass; then a mistake is planted in
the oracle (a dropped scale, a missing self edge, an unshifted softmax, ...)
and at least one pin must fail, so the pins are shown to see such mistakes.
"""
import numpy as np
import pytest

import oracle
from oracle import accept as oacc
from oracle import attention as oatt
from paper_2402_02082_gb300 import synth

import pins


# ----------------------------------------------------------------- attention
def test_single_key():
    pins.check_single_key(oracle.cross_attn)


def test_two_keys_closed_form():
    pins.check_two_keys_closed_form(oracle.cross_attn)


def test_cross_vs_sdpa():
    pins.check_cross_vs_sdpa(oracle.cross_attn)


def test_chain_is_causal():
    pins.check_chain_is_causal(oracle.tree_verify_attn)


def test_single_node_is_decode():
    pins.check_single_node_is_decode(oracle.tree_verify_attn)


def test_uniform_keys_mean():
    pins.check_uniform_keys_mean(oracle.tree_verify_attn)


def test_planted_key():
    pins.check_planted_key(oracle.cross_attn)


def test_prefix_permutation():
    pins.check_prefix_permutation(oracle.tree_verify_attn)


def test_tree_relabel():
    pins.check_tree_relabel(oracle.tree_verify_attn)


def test_cape_mask_golden():
    pins.check_cape_mask_golden(oracle.cape_mask, oracle.tree_allowed_mask)


def test_cape_mask_random():
    pins.check_cape_mask_random(oracle.cape_mask, oracle.tree_allowed_mask, synth.cape_tree)


def test_bf16_widening_exact():
    # bf16 bit patterns with known values: 1.0, -2.0, 0.5, smallest normal, 3.140625
    bits = np.array([0x3F80, 0xC000, 0x3F00, 0x0080, 0x4049], dtype=np.uint16)
    want = [1.0, -2.0, 0.5, 2.0 ** -126, 3.140625]
    assert list(oracle.widen(bits)) == want


def test_rows_beyond_tree_never_read():
    """Unused cache capacity (NaN here) must not reach any output."""
    w = synth.workload("tiny-f32")
    case = synth.make_case(w, garbage="nan")
    o1 = oracle.tree_verify_attn(case["q_tree"], case["parent_idx"], case["K"], case["V"], case["kv_len"])
    o2 = oracle.cross_attn(case["q_draft"][0], case["K"], case["V"], case["kv_len"])
    assert np.isfinite(o1).all() and np.isfinite(o2).all()


# ---------------------------------------------------------------- acceptance
def test_accept_golden():
    pins.check_accept_golden(oracle.tree_accept)


def test_accept_brute_force():
    pins.check_accept_brute_force(oracle.tree_accept)


def test_accept_chain_is_sd():
    pins.check_accept_chain_is_sd(oracle.tree_accept)


def test_accept_greedy_equivalence():
    pins.check_accept_greedy_equivalence(oracle.tree_accept)


def test_argmax_ties():
    pins.check_argmax_ties(oracle.row_argmax)


def test_accept_invariants_on_workloads():
    """Accepted path is a root chain whose every edge matches the target's argmax."""
    for w in synth.workloads():
        case = synth.make_case(w, with_kv=False)
        path, ln, bonus = oracle.tree_accept(case["draft_tokens"], case["parent_idx"], case["target_logits"])
        a = oracle.row_argmax(case["target_logits"])
        for b in range(w.B):
            p = [int(x) for x in path[b] if x >= 0]
            assert p[0] == 0 and len(p) == ln[b] + 1
            assert all(case["parent_idx"][b][p[k + 1]] == p[k] for k in range(len(p) - 1))
            assert all(case["draft_tokens"][b][p[k + 1]] == a[b][p[k]] for k in range(len(p) - 1))
            assert bonus[b] == a[b][p[-1]]


# ------------------------------------------------- planted mistakes must fail
def _expect_some_fail(checks):
    failed = 0
    for chk in checks:
        try:
            chk()
        except AssertionError:
            failed += 1
    assert failed > 0, "no pin noticed the planted mistake"


def test_mutant_missing_scale():
    bad = lambda q, K, V, L: oatt.cross_attn(q, K, V, L, scale=1.0)
    _expect_some_fail([lambda: pins.check_two_keys_closed_form(bad), lambda: pins.check_cross_vs_sdpa(bad)])


def test_mutant_k_v_swapped():
    bad = lambda q, K, V, L: oatt.cross_attn(q, V, K, L)
    _expect_some_fail([lambda: pins.check_cross_vs_sdpa(bad), lambda: pins.check_two_keys_closed_form(bad)])


def test_mutant_unshifted_softmax(monkeypatch):
    def unshifted(scores, allowed, values):
        s = np.where(allowed, scores, -np.inf)
        e = np.exp(s)
        return (e @ values) / e.sum(axis=1, keepdims=True)
    monkeypatch.setattr(oatt, "_softmax_rows_attend", unshifted)
    with np.errstate(all="ignore"):
        _expect_some_fail([lambda: pins.check_planted_key(oatt.cross_attn)])


def test_mutant_no_self_edge(monkeypatch):
    real = oatt.ancestors_or_self
    monkeypatch.setattr(oatt, "ancestors_or_self", lambda parent, i: real(parent, i)[1:])
    _expect_some_fail([lambda: pins.check_uniform_keys_mean(oatt.tree_verify_attn),
                       lambda: pins.check_chain_is_causal(oatt.tree_verify_attn)])


def test_mutant_parent_only(monkeypatch):
    monkeypatch.setattr(oatt, "ancestors_or_self",
                        lambda parent, i: [i] + ([int(parent[i])] if parent[i] >= 0 else []))
    _expect_some_fail([lambda: pins.check_uniform_keys_mean(oatt.tree_verify_attn),
                       lambda: pins.check_cape_mask_golden(oatt.cape_mask, oatt.tree_allowed_mask)])


def test_mutant_prefix_off_by_one(monkeypatch):
    real = oatt.tree_allowed_mask

    def short(parent, kv_len):
        m = real(parent, kv_len)
        if kv_len > 0:
            m[:, kv_len - 1] = False
        return m
    monkeypatch.setattr(oatt, "tree_allowed_mask", short)
    _expect_some_fail([lambda: pins.check_chain_is_causal(oatt.tree_verify_attn),
                       lambda: pins.check_single_node_is_decode(oatt.tree_verify_attn)])


def test_mutant_cape_mask_transposed():
    bad = lambda gamma, pos: oatt.cape_mask(gamma, pos).T
    _expect_some_fail([lambda: pins.check_cape_mask_golden(bad, oatt.tree_allowed_mask)])


def test_mutant_argmax_last_tie(monkeypatch):
    def last(lg):
        r = lg[..., ::-1]
        return (lg.shape[-1] - 1 - np.argmax(r, axis=-1)).astype(np.int32)
    monkeypatch.setattr(oacc, "row_argmax", last)
    _expect_some_fail([lambda: pins.check_argmax_ties(oacc.row_argmax),
                       lambda: pins.check_accept_brute_force(oacc.tree_accept)])


def test_mutant_accept_ignores_ancestors():
    def bad(draft, parent, lg):
        # accepts any node whose own edge matches, ignoring its ancestors
        B, n = draft.shape
        a = np.argmax(lg, axis=-1)
        path = np.full((B, n), -1, dtype=np.int32)
        ln = np.zeros(B, dtype=np.int32)
        bo = np.zeros(B, dtype=np.int32)
        for b in range(B):
            depth = [0] * n
            best = 0
            for c in range(1, n):
                depth[c] = depth[parent[b][c]] + 1
                if draft[b][c] == a[b][parent[b][c]] and depth[c] > depth[best]:
                    best = c
            chain = [best]
            while chain[-1] != 0:
                chain.append(int(parent[b][chain[-1]]))
            path[b, :len(chain)] = chain[::-1]
            ln[b] = depth[best]
            bo[b] = a[b][best]
        return path, ln, bo
    _expect_some_fail([lambda: pins.check_accept_brute_force(bad), lambda: pins.check_accept_golden(bad)])
