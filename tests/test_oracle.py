"""Pins of the fp64 oracle against what the mathematics fixes (no GPU).

Each test checks the oracle against something other than itself: hand-derived
closed forms (tests/golden), an independent library routine (torch's
scaled_dot_product_attention and softmax in fp64, scipy's logsumexp), invariants
(softmax rows sum to one; sink and recent positions are kept) or brute force
over all subsets on tiny inputs.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import logsumexp

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def rand(rng, *shape):
    return rng.standard_normal(shape)


# ----------------------------------------------------------------------------- golden closed forms

def test_golden_attention_basis():
    fx = load("attention_basis.json")
    o, lse = oracle.attention(np.array(fx["q"]), np.array(fx["keys"], float),
                              np.array(fx["values"], float), fx["scale"])
    np.testing.assert_allclose(o, fx["o"], atol=1e-14)
    assert abs(lse - fx["lse"]) < 1e-14


def test_golden_verify_causal():
    fx = load("verify_causal.json")
    keys = np.array(fx["keys"], float)[None, None]
    vals = np.array(fx["values"], float)[None, None]
    q = np.array(fx["q"], float)[None, None]
    o, lse = oracle.verify_attn(q, keys, vals, fx["t_ctx"])
    np.testing.assert_allclose(o[0, 0], fx["o"], atol=1e-14)
    np.testing.assert_allclose(lse[0, 0], fx["lse"], atol=1e-14)


def test_golden_window_scores():
    fx = load("window_scores_uniform.json")
    keys = np.array(fx["keys"], float)[None, None]
    qw = np.array(fx["q_win"], float)[None, None]
    lse = oracle.window_lse(qw, keys, fx["t_ctx"])
    np.testing.assert_allclose(lse[0, 0], fx["lse"], atol=1e-14)
    score = oracle.window_scores(qw, keys, lse, fx["t_ctx"])
    np.testing.assert_allclose(score[0, 0], fx["score"], atol=1e-14)


def test_golden_selection():
    fx = load("selection_example.json")
    score = np.array(fx["score"], float)
    for case in fx["cases"]:
        keep = oracle.select_from_scores(score, fx["t_ctx"], case["budget"], fx["n_sink"],
                                         fx["n_recent"], case["chunk"])
        assert keep.tolist() == case["keep"], case


def test_golden_boundary_score():
    """The tie band of every selection check is centred on this value: the score of the last
    middle position admitted, not the first one excluded, and nothing when no slot is ranked."""
    fx = load("boundary_example.json")
    score = np.array(fx["score"], float)
    for case in fx["cases"]:
        tau = oracle.boundary_score(score, fx["t_ctx"], case["budget"], fx["n_sink"], fx["n_recent"])
        assert tau == case["tau"], case
        if tau is not None:       # the kept middle is exactly the positions scoring at least tau
            keep = oracle.select_from_scores(score, fx["t_ctx"], case["budget"], fx["n_sink"], fx["n_recent"])
            mid = keep[(keep >= fx["n_sink"]) & (keep < fx["t_ctx"] - fx["n_recent"])]
            assert min(score[mid]) == tau


def test_golden_combine():
    fx = load("combine_two_halves.json")
    o, lse = oracle.combine(np.array(fx["o_part"]), np.array(fx["lse_part"]))
    np.testing.assert_allclose(o, fx["o"], atol=1e-14)
    np.testing.assert_allclose(lse, fx["lse"], atol=1e-14)


# ----------------------------------------------------------------------------- attention closed forms

def test_attention_identical_keys_gives_mean_value():
    rng = np.random.default_rng(1)
    k = np.tile(rand(rng, 1, 16), (9, 1))
    v = rand(rng, 9, 16)
    q = rand(rng, 16)
    o, lse = oracle.attention(q, k, v, 0.25)
    np.testing.assert_allclose(o, v.mean(axis=0), atol=1e-13)
    assert abs(lse - (0.25 * q @ k[0] + math.log(9))) < 1e-12


def test_attention_single_key_and_empty():
    rng = np.random.default_rng(2)
    k, v, q = rand(rng, 1, 8), rand(rng, 1, 8), rand(rng, 8)
    o, lse = oracle.attention(q, k, v, 0.5)
    np.testing.assert_allclose(o, v[0], atol=1e-15)
    assert abs(lse - 0.5 * q @ k[0]) < 1e-14
    o, lse = oracle.attention(q, np.zeros((0, 8)), np.zeros((0, 8)), 0.5)
    assert lse == -math.inf and not o.any()


def test_attention_one_hot_values_give_probabilities():
    rng = np.random.default_rng(3)
    m, d = 7, 32
    k, q = rand(rng, m, d), rand(rng, d)
    o, lse = oracle.attention(q, k, np.eye(m), 1 / math.sqrt(d))
    s = k @ q / math.sqrt(d)
    p = np.exp(s) / np.exp(s).sum()
    np.testing.assert_allclose(o, p, atol=1e-14)
    assert abs(o.sum() - 1) < 1e-13
    assert abs(lse - logsumexp(s)) < 1e-12


def test_attention_scale_invariance_of_shift():
    # adding the same vector c to every key shifts every logit by q.c: o unchanged, lse shifted
    rng = np.random.default_rng(4)
    k, v, q, c = rand(rng, 20, 16), rand(rng, 20, 16), rand(rng, 16), rand(rng, 16)
    o1, l1 = oracle.attention(q, k, v, 0.25)
    o2, l2 = oracle.attention(q, k + c, v, 0.25)
    np.testing.assert_allclose(o1, o2, atol=1e-12)
    assert abs((l2 - l1) - 0.25 * q @ c) < 1e-11


# ----------------------------------------------------------------------------- library cross-checks

def sdpa_reference(q, k, v, mask):
    """torch fp64 scaled_dot_product_attention with an explicit boolean mask."""
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q), torch.from_numpy(k), torch.from_numpy(v),
        attn_mask=torch.from_numpy(mask)).numpy()


@pytest.mark.parametrize("b,h_q,h_kv,d,t_ctx,n_q", [(2, 4, 2, 16, 37, 6), (1, 8, 2, 64, 130, 3),
                                                     (1, 2, 2, 8, 5, 1)])
def test_verify_matches_torch_sdpa(b, h_q, h_kv, d, t_ctx, n_q):
    rng = np.random.default_rng(5)
    t_cap = t_ctx + n_q + 2
    K, V = rand(rng, b, h_kv, t_cap, d), rand(rng, b, h_kv, t_cap, d)
    q = rand(rng, b, h_q, n_q, d)
    o, lse = oracle.verify_attn(q, K, V, t_ctx)
    g = h_q // h_kv
    Kx = np.repeat(K, g, axis=1)[:, :, : t_ctx + n_q]
    Vx = np.repeat(V, g, axis=1)[:, :, : t_ctx + n_q]
    mask = np.arange(t_ctx + n_q)[None, :] <= (t_ctx + np.arange(n_q))[:, None]
    ref = sdpa_reference(q, Kx, Vx, mask)
    np.testing.assert_allclose(o, ref, atol=1e-12)
    logits = np.einsum("bhid,bhkd->bhik", q, Kx) / math.sqrt(d)
    logits = np.where(mask, logits, -np.inf)
    np.testing.assert_allclose(lse, logsumexp(logits, axis=-1), atol=1e-12)


def test_verify_single_query_equals_decode():
    rng = np.random.default_rng(6)
    K, V = rand(rng, 1, 2, 50, 16), rand(rng, 1, 2, 50, 16)
    q = rand(rng, 1, 4, 1, 16)
    o, lse = oracle.verify_attn(q, K, V, 40)
    for h in range(4):
        oo, ll = oracle.attention(q[0, h, 0], K[0, h // 2, :41], V[0, h // 2, :41], 0.25)
        np.testing.assert_allclose(o[0, h, 0], oo, atol=1e-14)
        assert abs(lse[0, h, 0] - ll) < 1e-14


def test_window_lse_matches_logsumexp():
    rng = np.random.default_rng(7)
    b, h_q, h_kv, W, d, t = 2, 4, 2, 5, 8, 23
    K = rand(rng, b, h_kv, t + 3, d)
    qw = rand(rng, b, h_q, W, d)
    lse = oracle.window_lse(qw, K, t)
    for bi in range(b):
        for h in range(h_q):
            for w in range(W):
                p = t - W + w
                s = K[bi, h // 2, : p + 1] @ qw[bi, h, w] / math.sqrt(d)
                assert abs(lse[bi, h, w] - logsumexp(s)) < 1e-12


def test_window_scores_match_torch_softmax_and_sum_to_group_window():
    rng = np.random.default_rng(8)
    b, h_q, h_kv, W, d, t = 2, 8, 2, 6, 16, 40
    K = rand(rng, b, h_kv, t + 6, d)
    qw = rand(rng, b, h_q, W, d)
    lse = oracle.window_lse(qw, K, t)
    score = oracle.window_scores(qw, K, lse, t)
    g = h_q // h_kv
    # independent: torch softmax over the causal mask, summed over the group's heads and rows
    logits = torch.einsum("bhwd,bhkd->bhwk", torch.from_numpy(qw),
                          torch.from_numpy(np.repeat(K[:, :, :t], g, axis=1))) / math.sqrt(d)
    pos = torch.arange(t - W, t)
    mask = torch.arange(t)[None, :] <= pos[:, None]
    p = torch.softmax(logits.masked_fill(~mask, -math.inf), dim=-1)
    ref = p.reshape(b, h_kv, g, W, t).sum(dim=(2, 3)).numpy()
    np.testing.assert_allclose(score, ref, atol=1e-13)
    # every window row is a probability distribution over its prefix
    np.testing.assert_allclose(score.sum(axis=-1), g * W, rtol=1e-13)


# ----------------------------------------------------------------------------- combine

def test_combine_of_disjoint_parts_equals_union():
    rng = np.random.default_rng(9)
    m, d, rows = 60, 16, 3
    K, V = rand(rng, m, d), rand(rng, m, d)
    Q = rand(rng, rows, d)
    parts = np.array_split(rng.permutation(m), 4)
    parts.append(np.array([], dtype=int))          # an empty part is neutral
    o_part = np.zeros((len(parts), rows, d))
    lse_part = np.zeros((len(parts), rows))
    for s, idx in enumerate(parts):
        for r in range(rows):
            o_part[s, r], lse_part[s, r] = oracle.attention(Q[r], K[idx], V[idx], 0.25)
    o, lse = oracle.combine(o_part, lse_part)
    for r in range(rows):
        oo, ll = oracle.attention(Q[r], K, V, 0.25)
        np.testing.assert_allclose(o[r], oo, atol=1e-13)
        assert abs(lse[r] - ll) < 1e-12


def test_combine_all_empty():
    o, lse = oracle.combine(np.zeros((3, 2, 4)), np.full((3, 2), -np.inf))
    assert not o.any() and np.all(lse == -np.inf)


# ----------------------------------------------------------------------------- selection

def brute_force_keep(score, t_ctx, budget, n_sink, n_recent, chunk=1):
    """Best subset of middle positions (or chunks) by exhaustive enumeration.

    Among subsets of maximal total score, the lexicographically smallest sorted
    label tuple wins (that is what 'ties go to the lower index' means for a sum).
    """
    if budget >= t_ctx:
        return list(range(t_ctx))
    lo, hi = n_sink, t_ctx - n_recent
    free = budget - n_sink - n_recent
    if chunk == 1:
        labels = list(range(lo, hi))
        value = {p: score[p] for p in labels}
        members = {p: [p] for p in labels}
        k = free
    else:
        labels = list(range(lo // chunk, (hi - 1) // chunk + 1))
        members = {c: [p for p in range(c * chunk, c * chunk + chunk) if lo <= p < hi] for c in labels}
        value = {c: sum(score[p] for p in members[c]) for c in labels}
        k = free // chunk
    best, best_key = None, None
    for sub in itertools.combinations(labels, k):
        total = sum(value[c] for c in sub)
        key = (-total, sub)
        if best_key is None or key < best_key:
            best, best_key = sub, key
    chosen = [p for c in best for p in members[c]]
    return sorted(list(range(0, lo)) + chosen + list(range(hi, t_ctx)))


def test_selection_brute_force_integer_scores_with_ties():
    rng = np.random.default_rng(10)
    for trial in range(120):
        t = int(rng.integers(6, 15))
        n_sink = int(rng.integers(0, 3))
        n_recent = int(rng.integers(0, 4))
        if n_sink + n_recent >= t:
            continue
        budget = int(rng.integers(n_sink + n_recent, t + 2))
        chunk = int(rng.choice([1, 1, 2, 3]))
        score = rng.integers(0, 4, size=t).astype(float)     # many exact ties, exact sums
        keep = oracle.select_from_scores(score, t, budget, n_sink, n_recent, chunk)
        assert keep.tolist() == brute_force_keep(score, t, budget, n_sink, n_recent, chunk), \
            (trial, t, budget, n_sink, n_recent, chunk, score)


def test_selection_brute_force_real_scores():
    rng = np.random.default_rng(11)
    t, W, d = 14, 4, 8
    K = rand(rng, 1, 1, t + 2, d)
    qw = rand(rng, 1, 2, W, d)
    idx, count, score = oracle.select_budget(qw, K, t, budget=7, n_sink=1, n_recent=2)
    assert count[0, 0] == 7
    assert idx[0, 0].tolist() == brute_force_keep(score[0, 0], t, 7, 1, 2)


def test_selection_invariants_on_workload_shape():
    rng = np.random.default_rng(12)
    b, h_q, h_kv, W, d, t = 1, 4, 2, 32, 16, 300
    K = rand(rng, b, h_kv, t + 6, d)
    qw = rand(rng, b, h_q, W, d)
    for budget, n_sink, n_recent in [(64, 4, 16), (100, 0, 0), (40, 4, 36), (300, 4, 16), (512, 4, 16)]:
        idx, count, score = oracle.select_budget(qw, K, t, budget, n_sink, n_recent)
        for kv in range(h_kv):
            keep = idx[0, kv, : count[0, kv]]
            assert count[0, kv] == min(budget, t)
            assert np.all(np.diff(keep) > 0)                       # ascending, unique
            assert set(range(n_sink)) <= set(keep.tolist())
            assert set(range(t - n_recent, t)) <= set(keep.tolist())
            assert np.all(idx[0, kv, count[0, kv]:] == -1)
            tau = oracle.boundary_score(score[0, kv], t, budget, n_sink, n_recent)
            if tau is not None:
                mid = keep[(keep >= n_sink) & (keep < t - n_recent)]
                assert np.all(score[0, kv, mid] >= tau)
                out = np.setdiff1d(np.arange(n_sink, t - n_recent), mid)
                assert np.all(score[0, kv, out] <= tau)


def test_selection_all_equal_keys_takes_lowest_middle():
    t, W, d = 50, 4, 8
    K = np.ones((1, 1, t + 2, d))
    qw = np.random.default_rng(13).standard_normal((1, 1, W, d))
    idx, count, score = oracle.select_budget(qw, K, t, budget=12, n_sink=2, n_recent=3)
    # middle rows [2, 47) all tie below the window (which lies inside the recent rows)
    assert idx[0, 0, :12].tolist() == [0, 1, 2, 3, 4, 5, 6, 7, 8, 47, 48, 49]


def test_selection_monotone_in_planted_shift():
    rng = np.random.default_rng(14)
    t, W, d = 120, 8, 16
    K = rand(rng, 1, 1, t + 2, d)
    qw = rand(rng, 1, 1, W, d)
    u = qw[0, 0].sum(axis=0)
    u /= np.linalg.norm(u)
    base_idx, base_cnt, _ = oracle.select_budget(qw, K, t, budget=30, n_sink=2, n_recent=8)
    kept = base_idx[0, 0, : base_cnt[0, 0]]
    for p in kept[(kept >= 2) & (kept < t - 8)][:5]:
        K2 = K.copy()
        K2[0, 0, p] += 2.0 * u               # make key p more attended by the window
        idx2, cnt2, _ = oracle.select_budget(qw, K2, t, budget=30, n_sink=2, n_recent=8)
        assert p in idx2[0, 0, : cnt2[0, 0]]


def test_carried_lse_gives_same_selection():
    rng = np.random.default_rng(15)
    K = rand(rng, 2, 2, 90, 8)
    qw = rand(rng, 2, 4, 8, 8)
    lse = oracle.window_lse(qw, K, 84)
    a = oracle.select_budget(qw, K, 84, 30, 2, 10)
    b = oracle.select_budget(qw, K, 84, 30, 2, 10, lse_win=lse)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[2], b[2])


# ----------------------------------------------------------------------------- draft

def test_draft_with_full_budget_equals_full_attention():
    rng = np.random.default_rng(16)
    b, h_q, h_kv, d, t, gamma = 2, 4, 2, 16, 33, 4
    K, V = rand(rng, b, h_kv, t + gamma + 1, d), rand(rng, b, h_kv, t + gamma + 1, d)
    qw = rand(rng, b, h_q, 8, d)
    idx, count, _ = oracle.select_budget(qw, K, t, budget=64, n_sink=2, n_recent=4)
    assert np.all(count == t)
    for j in range(gamma):
        q = rand(rng, b, h_q, d)
        o, lse = oracle.draft_attn(q, K, V, idx, count, t, j)
        # the same query placed at position t + j of a verify block sees [0, t + j]
        q_blk = np.zeros((b, h_q, j + 1, d))
        q_blk[:, :, j] = q
        ov, lv = oracle.verify_attn(q_blk, K, V, t)
        np.testing.assert_allclose(o, ov[:, :, j], atol=1e-13)
        np.testing.assert_allclose(lse, lv[:, :, j], atol=1e-12)


def test_draft_matches_sdpa_over_gathered_rows():
    rng = np.random.default_rng(17)
    b, h_q, h_kv, d, t, budget = 1, 4, 2, 32, 64, 10
    K, V = rand(rng, b, h_kv, t + 6, d), rand(rng, b, h_kv, t + 6, d)
    idx = np.full((b, h_kv, budget), -1)
    count = np.array([[10, 7]])
    for kv in range(h_kv):
        idx[0, kv, : count[0, kv]] = np.sort(rng.choice(t, count[0, kv], replace=False))
    q = rand(rng, b, h_q, d)
    j = 2
    o, lse = oracle.draft_attn(q, K, V, idx, count, t, j)
    for h in range(h_q):
        kv = h // 2
        rows = np.concatenate([idx[0, kv, : count[0, kv]], np.arange(t, t + j + 1)])
        ref = sdpa_reference(q[0, h][None, None, None], K[0, kv, rows][None, None],
                             V[0, kv, rows][None, None], np.ones((1, rows.size), bool))
        np.testing.assert_allclose(o[0, h], ref[0, 0, 0], atol=1e-13)


# ----------------------------------------------------------------------------- one whole step

@pytest.mark.parametrize("budget", [7, 64])
def test_spec_step_against_independent_routines(budget):
    """The oracle's whole step (Algorithm 2: sparsify, gamma drafts, verify) against library
    routines and brute force: the view is the brute-force best subset of the torch-softmax
    scores, draft pass j is fp64 SDPA over the view plus rows t .. t+j with the j-th draft
    query, and the verify block is fp64 SDPA with the causal block mask."""
    rng = np.random.default_rng(18)
    b, h_q, h_kv, d, t, W, gamma, n_sink, n_recent = 1, 4, 2, 8, 13, 4, 3, 1, 2
    K, V = rand(rng, b, h_kv, t + gamma + 1, d), rand(rng, b, h_kv, t + gamma + 1, d)
    qw = rand(rng, b, h_q, W, d)
    qd = rand(rng, gamma, b, h_q, d)
    qv = rand(rng, b, h_q, gamma + 1, d)
    out = oracle.spec_step(K, V, qw, qd, qv, t, budget, n_sink, n_recent)
    g = h_q // h_kv
    logits = torch.einsum("bhwd,bhkd->bhwk", torch.from_numpy(qw),
                          torch.from_numpy(np.repeat(K[:, :, :t], g, axis=1))) / math.sqrt(d)
    mask = torch.arange(t)[None, :] <= torch.arange(t - W, t)[:, None]
    score = torch.softmax(logits.masked_fill(~mask, -math.inf), -1).reshape(b, h_kv, g, W, t).sum((2, 3)).numpy()
    np.testing.assert_allclose(out["score"], score, atol=1e-13)
    for kv in range(h_kv):
        keep = brute_force_keep(score[0, kv], t, budget, n_sink, n_recent) if budget < t else list(range(t))
        assert out["idx"][0, kv, : out["count"][0, kv]].tolist() == keep
        for j in range(gamma):
            rows = np.concatenate([np.array(keep, dtype=np.int64), np.arange(t, t + j + 1)])
            for h in range(kv * g, (kv + 1) * g):
                ref = sdpa_reference(qd[j, 0, h][None, None, None], K[0, kv, rows][None, None],
                                     V[0, kv, rows][None, None], np.ones((1, rows.size), bool))
                np.testing.assert_allclose(out["draft_o"][j, 0, h], ref[0, 0, 0], atol=1e-12)
                s = K[0, kv, rows] @ qd[j, 0, h] / math.sqrt(d)
                assert abs(out["draft_lse"][j, 0, h] - logsumexp(s)) < 1e-12
    Kx = np.repeat(K, g, axis=1)[:, :, : t + gamma + 1]
    Vx = np.repeat(V, g, axis=1)[:, :, : t + gamma + 1]
    vmask = np.arange(t + gamma + 1)[None, :] <= (t + np.arange(gamma + 1))[:, None]
    np.testing.assert_allclose(out["verify_o"], sdpa_reference(qv, Kx, Vx, vmask), atol=1e-12)
    vlog = np.where(vmask, np.einsum("bhid,bhkd->bhik", qv, Kx) / math.sqrt(d), -np.inf)
    np.testing.assert_allclose(out["verify_lse"], logsumexp(vlog, axis=-1), atol=1e-12)


def test_widen_bf16_bits_exact():
    x = torch.randn(1000).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.widen_bf16_bits(bits), x.double().numpy())


# ----------------------------------------------------------------------------- greedy acceptance

def test_golden_accept():
    fx = load("accept_examples.json")
    n, emit = oracle.accept_greedy(np.array(fx["draft"]), np.array(fx["verify"]))
    assert n.tolist() == fx["n_accept"]
    assert emit.tolist() == fx["emit"]


def test_golden_argmax_ties_and_nan():
    fx = load("argmax_ties.json")
    logits = np.array([[float(x) for x in row] for row in fx["logits"]])
    assert oracle.greedy_argmax(logits).tolist() == fx["argmax"]


def test_argmax_brute_force_with_ties_nan_and_signed_zero():
    # a plain scan over each row: the first strictly larger comparable value wins
    rng = np.random.default_rng(21)
    x = rng.integers(-3, 4, size=(400, 9)).astype(np.float32)
    x[rng.random(x.shape) < 0.15] = np.nan
    x[rng.random(x.shape) < 0.1] = -np.inf
    x[rng.random(x.shape) < 0.1] = -0.0
    x[::37] = np.nan
    x[5::11] = -np.inf                                  # rows whose numbers are all -inf ...
    x[5::22, ::2] = np.nan                              # ... some behind a leading NaN
    got = oracle.greedy_argmax(x)
    for r in range(x.shape[0]):
        best, best_id = None, 0
        for v in range(x.shape[1]):
            if not np.isnan(x[r, v]) and (best is None or x[r, v] > best):
                best, best_id = x[r, v], v
        assert got[r] == best_id, r


def test_accept_brute_force():
    rng = np.random.default_rng(22)
    for _ in range(200):
        gamma = int(rng.integers(1, 7))
        d = rng.integers(0, 3, size=(1, gamma))
        v = rng.integers(0, 3, size=(1, gamma + 1))
        n, emit = oracle.accept_greedy(d, v)
        # brute force: the largest k whose whole prefix agrees
        k = max(kk for kk in range(gamma + 1) if all(d[0, i] == v[0, i] for i in range(kk)))
        assert n[0] == k
        assert emit[0, :k].tolist() == d[0, :k].tolist() and emit[0, k] == v[0, k]
        assert np.all(emit[0, k + 1:] == -1)


# ----------------------------------------------------------------------------- cache update

def test_batch_advance_closed_cases():
    assert oracle.batch_advance(np.array([3, 1, 4]), n_q=6) == 2       # smallest k = 1 -> k + 1 rows
    assert oracle.batch_advance(np.array([5, 5]), n_q=6) == 6          # all drafts accepted
    assert oracle.batch_advance(np.array([0, 5]), n_q=6) == 1          # only the starting token settles
    assert oracle.batch_advance(np.array([9]), n_q=6) == 6             # clamped to the block


@pytest.mark.parametrize("window,advance", [(8, 3), (8, 6), (2, 3)])
def test_advance_window_equals_window_of_the_longer_context(window, advance):
    # the slid window must hold exactly the queries and causal LSEs a window taken at the
    # new length would have: compare with window_lse recomputed from scratch there
    rng = np.random.default_rng(31)
    b, hq, hkv, d, t, n_q = 2, 4, 2, 16, 40, 6
    K = rng.standard_normal((b, hkv, t + n_q, d))
    q_all = rng.standard_normal((b, hq, t + n_q, d))
    q_win = q_all[:, :, t - window: t]
    lse_win = oracle.window_lse(q_win, K, t)
    q_ver = q_all[:, :, t: t + n_q]
    _, lse_ver = oracle.verify_attn(q_ver, K, K, t)
    q_new, lse_new = oracle.advance_window(q_win, lse_win, q_ver, lse_ver, advance)
    t2 = t + advance
    assert np.array_equal(q_new, q_all[:, :, t2 - window: t2])
    np.testing.assert_allclose(lse_new, oracle.window_lse(q_all[:, :, t2 - window: t2], K, t2), rtol=0, atol=1e-12)


def test_append_view_closed_example():
    idx = np.array([[[0, 5, 9, -1, -1, -1]]])
    cnt = np.array([[3]])
    i2, c2, full = oracle.append_view(idx, cnt, t_ctx=12, advance=2, capacity=6)
    assert i2.tolist() == [[[0, 5, 9, 12, 13, -1]]] and c2.tolist() == [[5]] and not full
    i3, c3, full = oracle.append_view(i2, c2, t_ctx=14, advance=2, capacity=6)
    assert i3.tolist() == i2.tolist() and c3.tolist() == [[5]] and full     # no room: unchanged
