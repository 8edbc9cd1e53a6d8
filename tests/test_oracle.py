"""Pins for the CPU fp64 oracle (no GPU).

Each test checks the oracle against something other than itself: an
independent numpy brute force, a library routine for a special case
(torch SDPA for causal attention), closed forms, invariances the definition
implies, and the union-of-key-sets identity that the GPU split merge relies on.
"""
import math

import numpy as np
import pytest
import torch

from paper_2604_26412_gb300 import workloads as wl
from tests import brute, problems

CASES = [
    # (B, layers, lens, levels, tree, paged, page_size, hq, hkv, D)
    (1, 1, (20,), (1, 1, 1), False, False, 8, 4, 2, 4),
    (2, 1, (17, 5), (1, 1, 1, 1), False, True, 8, 4, 2, 8),
    (2, 1, (0, 9), (2, 2, 1), True, True, 8, 4, 1, 8),
    (1, 2, (15, 16), (3, 2, 1), True, False, 8, 8, 2, 4),
    (2, 2, (16, 3, 31, 1), (2, 3), True, True, 16, 4, 4, 128),
    (1, 1, (12,), (1, 1, 1, 1, 1, 1), False, True, 8, 8, 8, 128),
]


def _run_oracle(oracle_mod, p, scale=0.0):
    d = oracle_mod.make_desc(**p.desc_kwargs(scale))
    return oracle_mod.attn(d, p.q, p.tk, p.tv, p.page_table, p.seq_lens, p.dk, p.dv, p.tree_parent)


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("nq_mode", ["last", "all"])
def test_oracle_matches_brute_force(oracle_mod, case, nq_mode):
    B, layers, lens, levels, tree, paged, P, hq, hkv, D = case
    spec = problems.small_spec(B=B, layers=layers, lens=lens, levels=levels, tree=tree, paged=paged, page_size=P,
                               hq=hq, hkv=hkv, D=D, seed=3)
    N = spec.n_nodes
    p = problems.make(spec, n_query=(levels[-1] if nq_mode == "last" else N), seed=5)
    out, lse = _run_oracle(oracle_mod, p)
    bout, blse = brute.brute_attn(p.q, p.tk, p.tv, p.page_table, p.seq_lens, p.dk, p.dv, p.tree_parent,
                                  **p.brute_kwargs())
    np.testing.assert_allclose(out, bout, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, blse, rtol=0, atol=1e-12)


def test_oracle_scale_parameter(oracle_mod):
    spec = problems.small_spec(lens=(11,), levels=(2, 2), tree=True, hq=4, hkv=2, D=8, seed=9)
    p = problems.make(spec, seed=1)
    for scale in (1.0, 0.37):
        out, lse = _run_oracle(oracle_mod, p, scale)
        bout, blse = brute.brute_attn(p.q, p.tk, p.tv, p.page_table, p.seq_lens, p.dk, p.dv, p.tree_parent,
                                      **p.brute_kwargs(scale))
        np.testing.assert_allclose(out, bout, atol=1e-12)
        np.testing.assert_allclose(lse, blse, atol=1e-12)


def test_probabilities_sum_to_one_and_mask_is_exact(oracle_mod):
    spec = problems.small_spec(B=2, lens=(9, 14), levels=(3, 3, 2), tree=True, paged=True, page_size=8, hq=4,
                               hkv=2, D=8, seed=4)
    p = problems.make(spec, seed=2)
    d = oracle_mod.make_desc(**p.desc_kwargs())
    N = p.n_nodes
    for c in range(2):
        R = brute.reach_matrix(p.tree_parent[c])
        L = int(p.seq_lens[c])
        for nl in range(p.n_query):
            for h in range(4):
                pr = oracle_mod.attn_probs(d, p.q, p.tk, p.page_table, p.seq_lens, p.dk, p.tree_parent, c, nl, h)
                assert abs(pr.sum() - 1.0) < 1e-12
                n = N - p.n_query + nl
                vis = np.concatenate([np.ones(L, bool), R[n]])
                assert np.all(pr[~vis] == 0.0)
                assert np.all(pr[vis] > 0.0)


def test_equals_causal_attention_when_draft_is_next_tokens(oracle_mod):
    """Chain drafting whose draft KV are the next tokens == causal attention rows L..L+N-1."""
    L, N, hq, hkv, D = 13, 5, 8, 2, 16
    spec = problems.small_spec(lens=(L,), levels=(1,) * N, tree=False, paged=False, hq=hq, hkv=hkv, D=D, seed=6)
    p = problems.make(spec, seed=3)
    out, lse = _run_oracle(oracle_mod, p)
    # Full sequence = prefix followed by the draft tokens.
    K = np.concatenate([brute.bits_to_f64(p.tk[0, :, :L]), brute.bits_to_f64(p.dk[0, :, :N])], axis=1)
    V = np.concatenate([brute.bits_to_f64(p.tv[0, :, :L]), brute.bits_to_f64(p.dv[0, :, :N])], axis=1)
    G = hq // hkv
    Kt = torch.from_numpy(np.repeat(K, G, axis=0))[None]          # [1, hq, L+N, D]
    Vt = torch.from_numpy(np.repeat(V, G, axis=0))[None]
    # Queries of the draft rows placed at positions L..L+N-1; earlier rows are dummies.
    Q = np.zeros((hq, L + N, D))
    Q[:, L:] = brute.bits_to_f64(p.q[0]).transpose(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(Q)[None], Kt, Vt, is_causal=True)
    ref = ref[0, :, L:].numpy().transpose(1, 0, 2)                 # [N, hq, D]
    np.testing.assert_allclose(out[0], ref, atol=1e-12)
    # lse against an explicit log-sum-exp of the causal row.
    s = np.einsum("hnd,hkd->hnk", Q[:, L:], np.repeat(K, G, axis=0)) / math.sqrt(D)
    for n in range(N):
        row = s[:, n, :L + n + 1]
        np.testing.assert_allclose(lse[0, n], np.log(np.exp(row).sum(-1)), atol=1e-12)


def test_single_empty_draft_equals_last_causal_row(oracle_mod):
    """N = Nq = 1 with the query's own K/V as the only draft slot: the last causal row."""
    spec = problems.small_spec(lens=(10,), levels=(1,), tree=False, hq=4, hkv=2, D=8, seed=8)
    p = problems.make(spec, seed=4)
    out, _ = _run_oracle(oracle_mod, p)
    K = np.concatenate([brute.bits_to_f64(p.tk[0, :, :10]), brute.bits_to_f64(p.dk[0, :, :1])], axis=1)
    V = np.concatenate([brute.bits_to_f64(p.tv[0, :, :10]), brute.bits_to_f64(p.dv[0, :, :1])], axis=1)
    for h in range(4):
        q = brute.bits_to_f64(p.q[0, 0, h])
        s = K[h // 2] @ q / math.sqrt(8)
        w = np.exp(s - s.max())
        np.testing.assert_allclose(out[0, 0, h], (w / w.sum()) @ V[h // 2], atol=1e-12)


def test_page_permutation_invariance_and_paged_equals_contiguous(oracle_mod):
    spec = problems.small_spec(B=2, lens=(21, 9), levels=(2, 2), tree=True, paged=True, page_size=8, hq=4, hkv=2,
                               D=8, seed=12)
    p = problems.make(spec, seed=7)
    out0, lse0 = _run_oracle(oracle_mod, p)
    # Consistent shuffle of physical pages and table entries.
    rng = np.random.default_rng(0)
    perm = rng.permutation(p.num_pages)
    inv = np.argsort(perm)
    tk2, tv2 = p.tk[perm], p.tv[perm]           # new page i holds old page perm[i]
    table2 = p.page_table.copy()
    for c in range(2):
        npg = (int(p.seq_lens[c]) + 7) // 8
        table2[c, :npg] = inv[p.page_table[c, :npg]]
    p2 = problems.HostProblem(**{**p.__dict__, "tk": tk2, "tv": tv2, "page_table": table2})
    out1, lse1 = _run_oracle(oracle_mod, p2)
    assert np.array_equal(out0, out1) and np.array_equal(lse0, lse1)
    # Same prefix in a contiguous layout.
    l_cap = int(p.seq_lens.max())
    ctk = np.zeros((2, 2, l_cap, 8), np.uint16)
    ctv = np.zeros_like(ctk)
    for c in range(2):
        for j in range(int(p.seq_lens[c])):
            ctk[c, :, j] = p.tk[p.page_table[c, j // 8], :, j % 8]
            ctv[c, :, j] = p.tv[p.page_table[c, j // 8], :, j % 8]
    kw = p.desc_kwargs()
    kw.update(paged=False, page_size=0, max_pages_per_seq=0, num_pages=0, l_cap=l_cap)
    d = oracle_mod.make_desc(**kw)
    out2, lse2 = oracle_mod.attn(d, p.q, ctk, ctv, None, p.seq_lens, p.dk, p.dv, p.tree_parent)
    assert np.array_equal(out0, out2) and np.array_equal(lse0, lse2)


def test_width_one_tree_reduces_to_chain(oracle_mod):
    spec = problems.small_spec(B=2, lens=(7, 19), levels=(1,) * 6, tree=True, paged=True, page_size=8, hq=4, hkv=2,
                               D=8, seed=13)
    p = problems.make(spec, seed=8)
    assert np.array_equal(p.tree_parent[0], np.arange(-1, 5))
    out_t, lse_t = _run_oracle(oracle_mod, p)
    kw = p.desc_kwargs()
    kw["tree"] = False
    d = oracle_mod.make_desc(**kw)
    out_c, lse_c = oracle_mod.attn(d, p.q, p.tk, p.tv, p.page_table, p.seq_lens, p.dk, p.dv, None)
    assert np.array_equal(out_t, out_c) and np.array_equal(lse_t, lse_c)


def test_closed_forms(oracle_mod):
    # One visible key: L = 0, chain, query node 0 sees only slot 0.
    spec = problems.small_spec(lens=(0,), levels=(1,), tree=False, hq=2, hkv=1, D=8, seed=1)
    p = problems.make(spec, seed=1)
    out, lse = _run_oracle(oracle_mod, p)
    v = brute.bits_to_f64(p.dv[0, 0, 0])
    k = brute.bits_to_f64(p.dk[0, 0, 0])
    for h in range(2):
        np.testing.assert_array_equal(out[0, 0, h], v)
        s = brute.bits_to_f64(p.q[0, 0, h]) @ k / math.sqrt(8)
        assert abs(lse[0, 0, h] - s) < 1e-14
    # q = 0: uniform weights -> mean of visible V, lse = log(#visible).
    spec = problems.small_spec(B=1, lens=(13,), levels=(2, 2), tree=True, paged=True, page_size=8, hq=4, hkv=2, D=8,
                               seed=2)
    p = problems.make(spec, seed=2)
    p.q[:] = 0
    out, lse = _run_oracle(oracle_mod, p)
    R = brute.reach_matrix(p.tree_parent[0])
    for nl in range(p.n_query):
        n = p.n_nodes - p.n_query + nl
        for h in range(4):
            kv = h // 2
            rows = [brute.bits_to_f64(p.tv[p.page_table[0, j // 8], kv, j % 8]) for j in range(13)]
            rows += [brute.bits_to_f64(p.dv[0, kv, m]) for m in range(p.n_nodes) if R[n, m]]
            np.testing.assert_allclose(out[0, nl, h], np.mean(rows, axis=0), atol=1e-13)
            assert abs(lse[0, nl, h] - math.log(len(rows))) < 1e-13
    # scale -> tiny positive is the same as q = 0 in the limit; scale exactly 1e-300 gives uniform weights.
    p2 = problems.make(spec, seed=2)
    out_s, lse_s = _run_oracle(oracle_mod, p2, scale=1e-300)
    np.testing.assert_allclose(out_s, out, atol=1e-13)
    np.testing.assert_allclose(lse_s, lse, atol=1e-13)


def test_union_of_key_sets_merges_by_logaddexp(oracle_mod):
    """lse over A u B = log(e^lseA + e^lseB - e^lseD) where D = A n B (the draft part)."""
    L, L1 = 23, 9
    spec = problems.small_spec(lens=(L,), levels=(2, 2), tree=True, paged=False, hq=4, hkv=2, D=8, seed=21)
    p = problems.make(spec, seed=9)
    full_out, full_lse = _run_oracle(oracle_mod, p)

    def part(lo, hi):
        tk = np.ascontiguousarray(p.tk[:, :, lo:hi]) if hi > lo else np.zeros((1, 2, 1, 8), np.uint16)
        tv = np.ascontiguousarray(p.tv[:, :, lo:hi]) if hi > lo else np.zeros((1, 2, 1, 8), np.uint16)
        kw = p.desc_kwargs()
        kw["l_cap"] = max(hi - lo, 1)
        d = oracle_mod.make_desc(**kw)
        return oracle_mod.attn(d, p.q, tk, tv, None, np.array([hi - lo], np.int32), p.dk, p.dv, p.tree_parent)

    oa, la = part(0, L1)       # prefix[0:L1] + visible draft
    ob, lb = part(L1, L)       # prefix[L1:L] + visible draft
    od, ld = part(0, 0)        # visible draft only (counted twice above)
    m = np.maximum(np.maximum(la, lb), ld)
    wa, wb, wd = np.exp(la - m), np.exp(lb - m), np.exp(ld - m)
    lse = m + np.log(wa + wb - wd)
    out = (wa[..., None] * oa + wb[..., None] * ob - wd[..., None] * od) / (wa + wb - wd)[..., None]
    np.testing.assert_allclose(lse, full_lse, atol=1e-12)
    np.testing.assert_allclose(out, full_out, atol=1e-12)


def test_mask_probe_counts_visible_keys(oracle_mod):
    """q = 0 and one-hot V buckets: n_vis * out[d] counts visible keys in bucket d."""
    spec = problems.small_spec(B=2, lens=(37, 20), levels=(3, 4, 4), tree=True, paged=True, page_size=8, hq=4,
                               hkv=2, D=16, seed=17)
    p = problems.make(spec, seed=10)
    p.q[:] = 0
    one = 0x3F80  # bf16 1.0
    p.tv[:] = 0
    p.dv[:] = 0
    D = 16
    for c in range(2):
        for j in range(int(p.seq_lens[c])):
            p.tv[p.page_table[c, j // 8], :, j % 8, j % 12] = one        # prefix buckets 0..11
    for m in range(p.n_nodes):
        p.dv[:, :, m, 12 + m % 4] = one                                    # draft buckets 12..15
    out, lse = _run_oracle(oracle_mod, p)
    for c in range(2):
        R = brute.reach_matrix(p.tree_parent[c])
        L = int(p.seq_lens[c])
        for nl in range(p.n_query):
            n = p.n_nodes - p.n_query + nl
            expect = np.zeros(D)
            for j in range(L):
                expect[j % 12] += 1
            for m in range(p.n_nodes):
                if R[n, m]:
                    expect[12 + m % 4] += 1
            nvis = expect.sum()
            for h in range(4):
                np.testing.assert_allclose(out[c, nl, h] * nvis, expect, atol=1e-9)
                assert abs(lse[c, nl, h] - math.log(nvis)) < 1e-12


def test_oracle_rejects_invalid_inputs(oracle_mod):
    spec = problems.small_spec(B=1, lens=(9,), levels=(2, 2), tree=True, paged=True, page_size=8, hq=4, hkv=2, D=8)
    p = problems.make(spec, seed=1)
    d = oracle_mod.make_desc(**p.desc_kwargs())
    bad = p.tree_parent.copy()
    bad[0, 1] = 1  # a node cannot be its own parent
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.attn(d, p.q, p.tk, p.tv, p.page_table, p.seq_lens, p.dk, p.dv, bad)
    bad_pt = p.page_table.copy()
    bad_pt[0, 0] = p.num_pages
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.attn(d, p.q, p.tk, p.tv, bad_pt, p.seq_lens, p.dk, p.dv, p.tree_parent)
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.attn(d, p.q, p.tk, p.tv, p.page_table, np.array([10_000], np.int32), p.dk, p.dv, p.tree_parent)
