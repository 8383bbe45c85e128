"""Pins for the QER oracle (CoFiE Sec. 3.3, Eqs. 6-8), no GPU.

Eq. 6 against a brute-force loop on tiny inputs and against the equivalent
layout with every key head repeated per query head; Eq. 7 against closed
forms (identical tokens, duplicated or permuted text tokens, positive
scaling); Eq. 8 against its definition on special cases (rho = 0 and 1,
halfway counts, ties) and a planted-evidence stream; the score error bound
against honest rounding and a case that reaches it."""
import math

import numpy as np
import pytest

from oracle import qer_oracle as Q
from synth import qer as S


def _rand_bits(g, shape):
    return S.to_bf16_bits(g.standard_normal(shape).astype(np.float32))


def test_eq6_brute_force_loop():
    g = np.random.default_rng(1)
    n_text, H, H_kv, d, nv = 3, 4, 2, 5, 6
    q = _rand_bits(g, (n_text, H, d))
    k = _rand_bits(g, (nv, H_kv, d))
    qf, kf = Q.bf16_to_f64(q), Q.bf16_to_f64(k)
    a = Q.token_scores(q, k)
    for i in range(n_text):
        for j in range(nv):
            tot = 0.0
            for h in range(H):
                dot = 0.0
                for c in range(d):
                    dot += qf[i, h, c] * kf[j, h // (H // H_kv), c]
                tot += dot / math.sqrt(d)
            assert abs(a[i, j] - tot / H) <= 1e-12 * (1 + abs(tot))


def test_grouped_heads_equal_repeated_keys():
    g = np.random.default_rng(2)
    q = _rand_bits(g, (7, 8, 16))
    k = _rand_bits(g, (20, 2, 16))
    k_rep = np.repeat(k, 4, axis=1)  # key head h // 4 for query head h
    assert np.allclose(Q.token_scores(q, k), Q.token_scores(q, k_rep), rtol=0, atol=1e-12)


def test_identical_heads_reduce_to_one_dot_product():
    g = np.random.default_rng(3)
    q1 = _rand_bits(g, (5, 1, 32))
    k1 = _rand_bits(g, (9, 1, 32))
    a = Q.token_scores(np.repeat(q1, 6, axis=1), np.repeat(k1, 3, axis=1))
    want = (Q.bf16_to_f64(q1)[:, 0, :] @ Q.bf16_to_f64(k1)[:, 0, :].T) / math.sqrt(32)
    assert np.allclose(a, want, rtol=0, atol=1e-12)


def test_eq7_closed_forms():
    g = np.random.default_rng(4)
    q = _rand_bits(g, (6, 4, 8))
    tok = _rand_bits(g, (1, 2, 8))
    k = np.concatenate([np.repeat(tok, 5, axis=0), _rand_bits(g, (5, 2, 8))])
    w = Q.frame_relevance(Q.token_scores(q, k), 5)
    assert w[0] == pytest.approx(Q.token_scores(q, tok).max(), abs=1e-12)  # identical tokens
    perm = g.permutation(6)
    assert np.allclose(Q.frame_relevance(Q.token_scores(q[perm], k), 5), w, atol=1e-12)  # text order
    dup = np.concatenate([q, q[:2]])
    assert np.allclose(Q.frame_relevance(Q.token_scores(dup, k), 5), w, atol=1e-12)  # duplicated text
    # max over text, not mean: one text token aligned with every key dominates
    boost = np.concatenate([q, S.to_bf16_bits(np.repeat(Q.bf16_to_f64(tok).astype(np.float32), 2, axis=1) * 8)])
    w2 = Q.frame_relevance(Q.token_scores(boost, k), 5)
    assert w2[0] > w[0] and w2[0] == pytest.approx(Q.token_scores(boost[-1:], tok)[0, 0], rel=1e-12)


def test_eq8_special_cases():
    w = np.array([0.3, 0.9, 0.1, 0.9, 0.5])
    assert list(Q.select(w, 0.0)) == [1]                 # k = max(1, 0): the best frame
    assert list(Q.select(w, 1.0)) == [0, 1, 2, 3, 4]     # everything, chronological
    assert list(Q.select(w, 0.4)) == [1, 3]              # round(2.0) = 2; equal scores, both kept
    assert list(Q.select(w, 0.2)) == [1]                 # tie at the cut: the lower index wins
    assert Q.keep_count(5, 0.5) == 2 and Q.keep_count(7, 0.5) == 4  # 2.5 -> 2, 3.5 -> 4 (half to even)
    g = np.random.default_rng(5)
    for _ in range(50):
        m = int(g.integers(1, 40))
        w = g.random(m)
        rho = float(g.random())
        sel = Q.select(w, rho)
        assert len(sel) == max(1, round(rho * m)) and list(sel) == sorted(sel)
        rest = np.setdiff1d(np.arange(m), sel)
        if len(rest):
            assert w[sel].min() >= w[rest].max()


def test_planted_evidence_ranks_first():
    spec = S.QerSpec(n_text=32, n_frames=24, tokens_per_frame=16, n_evidence=3, seed=11)
    q, k, ev = S.generate(spec)
    w, sel = Q.run(q, k, spec.tokens_per_frame, rho=3 / 24)
    assert list(sel) == list(ev)


def test_score_bound_covers_bf16_group_sums():
    """The bound admits the error of an honest bf16 group-sum + fp32 path."""
    spec = S.QerSpec(n_text=16, n_frames=3, tokens_per_frame=8, seed=12)
    q, k, _ = S.generate(spec)
    qf = Q.bf16_to_f64(q).reshape(16, 8, 4, 128).sum(axis=2)            # head groups
    qg = S.to_bf16_bits(qf.astype(np.float32))                           # rounded to bf16
    kf = Q.bf16_to_f64(k)
    approx = np.einsum("igd,jgd->ij", Q.bf16_to_f64(qg).astype(np.float32), kf.astype(np.float32),
                       dtype=np.float32).astype(np.float64) / (32 * np.sqrt(128))
    w_approx = approx.max(axis=0).reshape(-1, 8).mean(axis=1)
    w, _ = Q.run(q, k, 8, 0.5)
    assert np.all(np.abs(w_approx - w) <= Q.score_bound(q, k, 8))


def test_score_bound_reached_by_a_rounding_worst_case():
    """Two query heads in one group, 1 and 2^-8 in every component, sum to
    1 + 2^-8, halfway between two bf16 values: the group sum rounds to 1 (half
    to even) and every product has the same sign, so the error is the whole
    2^-8 relative term: w = 1 + 2^-8 exactly, the group-sum path gives 1."""
    d = 4
    q = np.zeros((1, 2, d), dtype=np.float32)
    q[:, 0, :], q[:, 1, :] = 1.0, 2.0 ** -8
    q_bits = S.to_bf16_bits(q)
    k_bits = S.to_bf16_bits(np.ones((3, 1, d), dtype=np.float32))
    qg = Q.bf16_to_f64(S.to_bf16_bits(Q.bf16_to_f64(q_bits).sum(axis=1).astype(np.float32)))
    assert qg[0, 0] == 1.0
    w_group = (qg @ Q.bf16_to_f64(k_bits)[:, 0, :].T / (2 * np.sqrt(d))).max(axis=0).mean()
    w, _ = Q.run(q_bits, k_bits, 3, 1.0)
    assert w[0] == 1 + 2.0 ** -8 and w_group == 1.0
    bound = Q.score_bound(q_bits, k_bits, 3)[0]
    assert bound >= w[0] - w_group >= 0.99 * bound
