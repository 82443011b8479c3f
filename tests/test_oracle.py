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


# ----------------------------------------------------------- CaPE expansion
from oracle import cape as ocape
from oracle import kvcache as okv


def test_cape_expand_golden():
    pins.check_cape_expand_golden(ocape.cape_expand, ocape.expansion_size)


def test_cape_expand_brute_force():
    pins.check_cape_expand_brute_force(ocape.cape_expand, ocape.expansion_size)


def test_cape_expand_mask():
    pins.check_cape_expand_mask(ocape.cape_expand, oracle.cape_mask, oracle.tree_allowed_mask)


def test_cape_expand_cap():
    pins.check_cape_expand_cap(ocape.cape_expand)


def _cape_pins():
    return [lambda: pins.check_cape_expand_golden(ocape.cape_expand, ocape.expansion_size),
            lambda: pins.check_cape_expand_brute_force(ocape.cape_expand, ocape.expansion_size),
            lambda: pins.check_cape_expand_mask(ocape.cape_expand, oracle.cape_mask,
                                                oracle.tree_allowed_mask),
            lambda: pins.check_cape_expand_cap(ocape.cape_expand)]


def test_mutant_s_thresholds_in_fp32(monkeypatch):
    # comparing with the thresholds rounded to binary32 (p <= 0.3f) puts
    # 0.3f = 0.3000000119... in the first bucket
    def fp32_thresholds(p):
        x = np.float32(p)
        for upper, k in ocape._S_TABLE:
            if x <= np.float32(float(upper)):
                return k
        return ocape._S_LAST
    monkeypatch.setattr(ocape, "expansion_size", fp32_thresholds)
    _expect_some_fail(_cape_pins())


def test_mutant_set_keeps_proposal_token(monkeypatch):
    monkeypatch.setattr(ocape, "expansion_set", lambda order, k: order[0:k])
    _expect_some_fail(_cape_pins())


def test_mutant_ties_to_higher_id(monkeypatch):
    def ranked(row):
        vals = [float(v) + 0.0 for v in row]
        return sorted(range(len(vals)), key=lambda t: (-vals[t], -t))
    monkeypatch.setattr(ocape, "ranked_tokens", ranked)
    _expect_some_fail(_cape_pins())


def test_mutant_cap_cuts_linearized_tail(monkeypatch):
    monkeypatch.setattr(ocape, "keep_after_cap",
                        lambda cands, room: sorted(cands, key=lambda c: (c[1], c[2]))[:room])
    _expect_some_fail(_cape_pins())


def test_mutant_expansion_under_proposal_token(monkeypatch):
    real = ocape.cape_expand

    def bad(probs, root, max_tokens=32, fixed_k=None):
        tok, par, nn, conf, ku = real(probs, root, max_tokens, fixed_k)
        gamma = probs.shape[1]
        for b in range(len(nn)):
            par[b, gamma + 1:nn[b]] += 1          # child of x_{t+i} instead of its sibling
        return tok, par, nn, conf, ku
    monkeypatch.setattr(ocape, "cape_expand", bad)
    _expect_some_fail(_cape_pins())


# --------------------------------------------------------- KV-cache update
def test_kv_compact_golden():
    pins.check_kv_compact_golden(okv.kv_compact)


def test_kv_compact_attention():
    pins.check_kv_compact_attention(okv.kv_compact, oracle.tree_verify_attn, oracle.cross_attn)


def test_kv_compact_chain_identity():
    pins.check_kv_compact_chain_identity(okv.kv_compact)


def _kv_pins(fn):
    return [lambda: pins.check_kv_compact_golden(fn),
            lambda: pins.check_kv_compact_attention(fn, oracle.tree_verify_attn, oracle.cross_attn),
            lambda: pins.check_kv_compact_chain_identity(fn)]


def test_mutant_kv_length_without_root():
    def bad(K, V, kv_len, path, length):
        K2, V2, nl = okv.kv_compact(K, V, kv_len, path, length)
        return K2, V2, nl - 1
    _expect_some_fail(_kv_pins(bad))


def test_mutant_kv_skips_root_entry():
    def bad(K, V, kv_len, path, length):
        shifted = np.concatenate([path[:, 1:], np.full((path.shape[0], 1), -1, path.dtype)], axis=1)
        shifted[shifted < 0] = 0
        return okv.kv_compact(K, V, kv_len, shifted, length)
    _expect_some_fail(_kv_pins(bad))


def test_mutant_kv_reversed_path():
    def bad(K, V, kv_len, path, length):
        rev = path.copy()
        for b in range(path.shape[0]):
            m = int(length[b]) + 1
            rev[b, :m] = path[b, :m][::-1]
        return okv.kv_compact(K, V, kv_len, rev, length)
    _expect_some_fail(_kv_pins(bad))


# ------------------------------------------------- speculative sampling
from oracle import sampling as osamp


def test_spec_sample_golden():
    pins.check_spec_sample_golden(osamp.spec_sample_accept)


def test_spec_sample_is_target_sampling():
    pins.check_spec_sample_is_target_sampling(osamp.spec_sample_accept)


def test_spec_sample_same_model_accepts():
    pins.check_spec_sample_same_model_accepts(osamp.spec_sample_accept)


def _sampling_pins():
    return [lambda: pins.check_spec_sample_golden(osamp.spec_sample_accept),
            lambda: pins.check_spec_sample_is_target_sampling(osamp.spec_sample_accept),
            lambda: pins.check_spec_sample_same_model_accepts(osamp.spec_sample_accept)]


def test_mutant_sampling_ratio_inverted(monkeypatch):
    monkeypatch.setattr(osamp, "accepts", lambda u, pd, pt: float(u) * float(pt) < float(pd))
    _expect_some_fail(_sampling_pins())


def test_mutant_sampling_non_strict(monkeypatch):
    monkeypatch.setattr(osamp, "accepts", lambda u, pd, pt: float(u) * float(pd) <= float(pt))
    _expect_some_fail(_sampling_pins())


def test_mutant_sampling_unclipped_residual(monkeypatch):
    def unclipped(pt, pd):
        w = pt - pd.astype(np.float64)
        return w if w.sum() > 0 else pt
    monkeypatch.setattr(osamp, "residual_weights", unclipped)
    _expect_some_fail(_sampling_pins())


def test_mutant_sampling_unnormalised_draw(monkeypatch):
    def raw(w, v):
        c = np.cumsum(w)
        idx = int(np.searchsorted(c, float(v), side="right"))
        return min(idx, len(w) - 1)
    monkeypatch.setattr(osamp, "inverse_cdf", raw)
    _expect_some_fail(_sampling_pins())


def test_mutant_sampling_bonus_from_last_proposal_row():
    def bad(draft_tokens, draft_probs, target_logits, uniforms):
        # the extra token after a full acceptance drawn from p_T,gamma (the last
        # proposal position) instead of p_T,gamma+1
        shifted = target_logits.copy()
        shifted[:, -1] = target_logits[:, -2]
        n, tok = osamp.spec_sample_accept(draft_tokens, draft_probs, target_logits, uniforms)
        n2, tok2 = osamp.spec_sample_accept(draft_tokens, draft_probs, shifted, uniforms)
        gamma = draft_tokens.shape[1]
        return n, np.where(n == gamma, tok2, tok)
    _expect_some_fail([lambda: pins.check_spec_sample_golden(bad),
                       lambda: pins.check_spec_sample_same_model_accepts(bad)])


# ------------------------------------------------ grouped-query attention
def test_gqa_is_repeated_kv():
    pins.check_gqa_is_repeated_kv(oracle.cross_attn, oracle.tree_verify_attn)


def test_mutant_gqa_interleaved_heads(monkeypatch):
    # query head h reading cached head h % H_kv (interleaved) instead of its group's
    monkeypatch.setattr(oatt, "kv_head", lambda h, H, H_kv: h % H_kv)
    _expect_some_fail([lambda: pins.check_gqa_is_repeated_kv(oracle.cross_attn, oracle.tree_verify_attn)])


# --------------------------------------------- training-time block mask
def test_block_mask_golden():
    pins.check_block_mask_golden(oatt.block_mask)


def test_block_attn_is_delayed_cross():
    pins.check_block_attn_is_delayed_cross(oatt.block_cross_attn, oracle.cross_attn)


def test_mutant_block_mask_inclusive(monkeypatch):
    # a position also seeing its own block (block(j) >= block(k))
    monkeypatch.setattr(oatt, "block_mask",
                        lambda T, L: (np.arange(T) // L)[:, None] >= (np.arange(T) // L)[None, :])
    _expect_some_fail([lambda: pins.check_block_mask_golden(oatt.block_mask),
                       lambda: pins.check_block_attn_is_delayed_cross(oatt.block_cross_attn, oracle.cross_attn)])


def test_mutant_block_mask_causal(monkeypatch):
    # a plain causal mask (k < j) instead of whole earlier blocks
    monkeypatch.setattr(oatt, "block_mask", lambda T, L: np.tril(np.ones((T, T), dtype=bool), -1))
    _expect_some_fail([lambda: pins.check_block_mask_golden(oatt.block_mask),
                       lambda: pins.check_block_attn_is_delayed_cross(oatt.block_cross_attn, oracle.cross_attn)])
