"""Plain fp64 CPU oracle for the KV-cache attention of one BudgetDraft speculative step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import or call this
module: only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py`` use it.  It shares no code with the CUDA path.

Every function is the plain definition of what the step computes, written with
numpy in float64.  Inputs are the bf16 values the kernels see, widened exactly to
float64 by the caller.  Nothing here is blocked, fused or reordered: a reader
can check each function against the paper by eye.

Paper references (BudgetDraft, arXiv 2606.00144):
  * Sparse drafter view K_S^sp(B) selected from the drafter prefix cache under a
    KV budget B: Sec. 3.1 (Eq. p_S) and the TopKChunks construction of Sec. 3.4
    (the prefix is cut into chunks of s positions, each chunk is ranked by the
    attention weight it accumulates, and the best floor(B/s) chunks are kept), which
    Algorithm 1 and the sparsify step of Algorithm 2 both use.
  * Draft step: gamma autoregressive drafter steps over K_S^sp(B) (Algorithm 2,
    Draft; Sec. 3.5).
  * Verify step: the verifier checks all gamma drafts in one forward over the
    full cache K_L^full (Algorithm 2, Verify; Sec. 3.5).
  * Cache update: accepted tokens are appended to both caches (Algorithm 2,
    Update), which is why the drafter's own new rows join its sparse view.

Readings where the paper is silent:
  * softmax scale 1/sqrt(d), no soft-cap; caches hold post-RoPE keys, so a row
    gathered by index keeps its position (Sec. 3.4, explicit position IDs);
  * "cumulative attention weight" of key k = sum over the GQA group's heads and
    over a window of the last W context queries of their causal softmax
    probability on k (token level, s = 1, with sink and recent positions always
    kept, as the graded workloads specify); ties at the budget boundary go to
    the lower position; the kept set is returned in ascending order;
  * chunk level (s > 1): chunks are aligned at multiples of s from position 0,
    a chunk's score is the sum of its middle members' scores, ties go to the
    lower chunk; the sink/recent rule is the same;
  * query i of a verify block sits at position t_ctx + i and sees keys
    [0, t_ctx + i]; draft pass j sees the selected rows plus its own rows
    t_ctx .. t_ctx + j.

Pins (tests/test_oracle.py, CPU; none of this module is "parity unpinned"):
  * attention: hand-derived basis fixture, identical keys -> mean value, one-hot
    values -> the probabilities, shift invariance, single and empty key sets;
  * verify_attn: hand-derived causal fixture, torch fp64 SDPA with a causal block
    mask, one query = decode over the prefix;
  * draft_attn: torch fp64 SDPA over the gathered rows, full budget = full attention;
  * window_lse / window_scores (and window_positions): scipy logsumexp, torch softmax,
    scores summing to G * W, a hand-derived uniform fixture;
  * select_from_scores / select_budget (and topk_lower_index): exhaustive subset
    enumeration with integer and real scores and ties (token and chunk level), all
    equal keys, monotonicity in a planted shift, carried LSE = recomputed LSE;
  * boundary_score: a fixture whose last admitted and first excluded scores differ;
  * combine: a hand-derived fixture, disjoint parts = union, all parts empty;
  * spec_step: brute-force selection over torch-softmax scores and fp64 SDPA;
  * greedy_argmax / accept_greedy: fixtures and brute force with ties, NaN, signed
    zeros; batch_advance / advance_window / append_view: closed cases and the window
    of the longer context; widen_bf16_bits: exact against torch's bf16 widening.
"""

from __future__ import annotations

import math

import numpy as np

NEG_INF = float("-inf")


# ---------------------------------------------------------------------------
# Attention by definition (Sec. 3.1: the drafter's p_S over K_S^sp(B) and the
# verifier's p_L over K_L^full are both ordinary softmax attention).
# ---------------------------------------------------------------------------

def attention(q: np.ndarray, keys: np.ndarray, values: np.ndarray, scale: float):
    """Softmax attention of one query over a set of key/value rows.

    q: [d]; keys, values: [m, d] (float64).  Returns (o [d], lse) with
        s_k = scale * (q . k_k),  lse = log sum_k exp(s_k),
        o = sum_k exp(s_k - lse) v_k.
    An empty key set gives o = 0 and lse = -inf (the neutral element of the
    log-sum-exp merge below).
    """
    q = np.asarray(q, dtype=np.float64)
    keys = np.asarray(keys, dtype=np.float64)
    values = np.asarray(values, dtype=np.float64)
    if keys.shape[0] == 0:
        return np.zeros(values.shape[1], dtype=np.float64), NEG_INF
    s = scale * (keys @ q)
    m = s.max()
    e = np.exp(s - m)
    l = e.sum()
    o = (e @ values) / l
    return o, m + math.log(l)


def combine(o_part: np.ndarray, lse_part: np.ndarray):
    """Merge attention results computed over disjoint key sets.

    o_part: [n, rows, d], each row normalised over its own key set;
    lse_part: [n, rows].  With L = log sum_s exp(lse_s), the merged row is
    sum_s exp(lse_s - L) o_s, which equals attention over the union of the key
    sets.  Rows whose parts are all empty give o = 0, L = -inf.
    """
    o_part = np.asarray(o_part, dtype=np.float64)
    lse_part = np.asarray(lse_part, dtype=np.float64)
    n, rows, d = o_part.shape
    o = np.zeros((rows, d), dtype=np.float64)
    lse = np.full(rows, NEG_INF, dtype=np.float64)
    for r in range(rows):
        finite = np.isfinite(lse_part[:, r])
        if not finite.any():
            continue
        m = lse_part[finite, r].max()
        w = np.exp(lse_part[finite, r] - m)
        L = m + math.log(w.sum())
        lse[r] = L
        o[r] = (np.exp(lse_part[finite, r] - L)[:, None] * o_part[finite, r, :]).sum(axis=0)
    return o, lse


# ---------------------------------------------------------------------------
# Verify step (Algorithm 2, Verify): n_q = gamma + 1 queries over the full cache
# with a causal mask inside the block.
# ---------------------------------------------------------------------------

def verify_attn(q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray, t_ctx: int):
    """q: [b, h_q, n_q, d]; caches: [b, h_kv, t_cap, d].

    Query i of head h sits at position t_ctx + i and attends to keys
    [0, t_ctx + i] of KV head h // (h_q / h_kv).  Returns o [b, h_q, n_q, d]
    and lse [b, h_q, n_q].
    """
    b, h_q, n_q, d = q.shape
    h_kv = k_cache.shape[1]
    group = h_q // h_kv
    scale = 1.0 / math.sqrt(d)
    o = np.zeros((b, h_q, n_q, d), dtype=np.float64)
    lse = np.zeros((b, h_q, n_q), dtype=np.float64)
    for bi in range(b):
        for h in range(h_q):
            kv = h // group
            keys = k_cache[bi, kv, : t_ctx + n_q]
            vals = v_cache[bi, kv, : t_ctx + n_q]
            logits = scale * (q[bi, h] @ keys.T)          # [n_q, t_ctx + n_q]
            for i in range(n_q):
                s = logits[i, : t_ctx + i + 1]             # causal: keys [0, t_ctx + i]
                m = s.max()
                e = np.exp(s - m)
                l = e.sum()
                o[bi, h, i] = (e @ vals[: t_ctx + i + 1]) / l
                lse[bi, h, i] = m + math.log(l)
    return o, lse


# ---------------------------------------------------------------------------
# Draft step (Algorithm 2, Draft): pass j of the gamma drafter passes, one query
# per head over the sparse view plus the drafter's own new rows.
# ---------------------------------------------------------------------------

def draft_attn(q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray,
               idx: np.ndarray, count: np.ndarray, t_ctx: int, step_j: int):
    """q: [b, h_q, d]; idx: [b, h_kv, budget] (positions); count: [b, h_kv].

    Pass j attends to rows idx[b, kv, :count[b, kv]] together with rows
    t_ctx .. t_ctx + step_j (the tokens drafted so far, own row included).
    Returns o [b, h_q, d], lse [b, h_q].
    """
    b, h_q, d = q.shape
    h_kv = k_cache.shape[1]
    group = h_q // h_kv
    scale = 1.0 / math.sqrt(d)
    o = np.zeros((b, h_q, d), dtype=np.float64)
    lse = np.zeros((b, h_q), dtype=np.float64)
    for bi in range(b):
        for h in range(h_q):
            kv = h // group
            rows = list(idx[bi, kv, : int(count[bi, kv])]) + list(range(t_ctx, t_ctx + step_j + 1))
            rows = np.asarray(rows, dtype=np.int64)
            o[bi, h], lse[bi, h] = attention(q[bi, h], k_cache[bi, kv, rows], v_cache[bi, kv, rows], scale)
    return o, lse


# ---------------------------------------------------------------------------
# Budget selection (Sec. 3.4 TopKChunks; Algorithm 2, sparsify).
# ---------------------------------------------------------------------------

def window_positions(t_ctx: int, window: int) -> np.ndarray:
    """Positions of the observation window: the last W context positions."""
    return np.arange(t_ctx - window, t_ctx, dtype=np.int64)


def window_lse(q_win: np.ndarray, k_cache: np.ndarray, t_ctx: int):
    """Softmax normaliser of each window query over its causal prefix.

    q_win: [b, h_q, W, d]; window row w sits at p_w = t_ctx - W + w and
    attends to keys [0, p_w].  Returns lse [b, h_q, W].
    """
    b, h_q, window, d = q_win.shape
    h_kv = k_cache.shape[1]
    group = h_q // h_kv
    scale = 1.0 / math.sqrt(d)
    pos = window_positions(t_ctx, window)
    lse = np.zeros((b, h_q, window), dtype=np.float64)
    for bi in range(b):
        for h in range(h_q):
            kv = h // group
            logits = scale * (q_win[bi, h] @ k_cache[bi, kv, :t_ctx].T)     # [W, t_ctx]
            for w in range(window):
                s = logits[w, : pos[w] + 1]
                m = s.max()
                lse[bi, h, w] = m + math.log(np.exp(s - m).sum())
    return lse


def window_scores(q_win: np.ndarray, k_cache: np.ndarray, lse_win: np.ndarray, t_ctx: int):
    """Cumulative attention weight of every context key, pooled over the group.

    score[b, kv, k] = sum over heads h of group kv and window rows w with
    k <= p_w of exp(scale * q_{h,w} . k_k - lse_{h,w}), i.e. the sum of the
    window rows' softmax probabilities on key k.  Returns [b, h_kv, t_ctx].
    """
    b, h_q, window, d = q_win.shape
    h_kv = k_cache.shape[1]
    group = h_q // h_kv
    scale = 1.0 / math.sqrt(d)
    pos = window_positions(t_ctx, window)
    causal = np.arange(t_ctx)[None, :] <= pos[:, None]                  # [W, t_ctx]
    score = np.zeros((b, h_kv, t_ctx), dtype=np.float64)
    for bi in range(b):
        for kv in range(h_kv):
            keys = k_cache[bi, kv, :t_ctx]
            for g in range(group):
                h = kv * group + g
                p = np.exp(scale * (q_win[bi, h] @ keys.T) - lse_win[bi, h][:, None])   # [W, t_ctx]
                p[~causal] = 0.0                                  # row w sees [0, p_w]
                score[bi, kv] += p.sum(axis=0)
    return score


def topk_lower_index(values: np.ndarray, labels: np.ndarray, k: int) -> np.ndarray:
    """The k labels with the largest values; equal values prefer the lower label."""
    order = np.lexsort((labels, -values))        # primary: value desc, then label asc
    return labels[order[:k]]


def select_from_scores(score: np.ndarray, t_ctx: int, budget: int, n_sink: int,
                       n_recent: int, chunk: int = 1) -> np.ndarray:
    """Kept positions of one (sequence, KV head), ascending.

    score: [t_ctx] cumulative attention weights.  If budget >= t_ctx every
    position is kept.  Otherwise keep the sinks [0, n_sink), the recent
    positions [t_ctx - n_recent, t_ctx) and, from the middle
    [n_sink, t_ctx - n_recent):
      * chunk == 1: the top (budget - n_sink - n_recent) positions by score;
      * chunk == s > 1: the top floor((budget - n_sink - n_recent) / s) chunks
        (chunk c covers positions [c s, c s + s) intersected with the middle),
        a chunk scored by the sum of its members' scores.
    Ties go to the lower position (lower chunk).
    """
    if budget >= t_ctx:
        return np.arange(t_ctx, dtype=np.int64)
    lo, hi = n_sink, t_ctx - n_recent
    mid = np.arange(lo, hi, dtype=np.int64)
    free = budget - n_sink - n_recent
    if chunk == 1:
        chosen = topk_lower_index(score[lo:hi], mid, free)
    else:
        first, last = lo // chunk, (hi - 1) // chunk
        chunk_ids = np.arange(first, last + 1, dtype=np.int64)
        chunk_score = np.array([score[max(c * chunk, lo): min(c * chunk + chunk, hi)].sum()
                                for c in chunk_ids])
        top = topk_lower_index(chunk_score, chunk_ids, free // chunk)
        chosen = np.concatenate([np.arange(max(c * chunk, lo), min(c * chunk + chunk, hi))
                                 for c in top] + [np.zeros(0, dtype=np.int64)])
    keep = np.concatenate([np.arange(0, lo), chosen, np.arange(hi, t_ctx)]).astype(np.int64)
    return np.sort(keep)


def select_budget(q_win: np.ndarray, k_cache: np.ndarray, t_ctx: int, budget: int,
                  n_sink: int, n_recent: int, chunk: int = 1, lse_win: np.ndarray | None = None):
    """Sparse drafter view K_S^sp(B) of every (sequence, KV head).

    Returns (idx [b, h_kv, budget] int64 padded with -1, count [b, h_kv],
    score [b, h_kv, t_ctx]).  lse_win defaults to the oracle's own window_lse.
    """
    b, h_q, window, d = q_win.shape
    h_kv = k_cache.shape[1]
    if lse_win is None:
        lse_win = window_lse(q_win, k_cache, t_ctx)
    score = window_scores(q_win, k_cache, lse_win, t_ctx)
    idx = np.full((b, h_kv, budget), -1, dtype=np.int64)
    count = np.zeros((b, h_kv), dtype=np.int64)
    for bi in range(b):
        for kv in range(h_kv):
            keep = select_from_scores(score[bi, kv], t_ctx, budget, n_sink, n_recent, chunk)
            idx[bi, kv, : keep.size] = keep
            count[bi, kv] = keep.size
    return idx, count, score


def boundary_score(score_row: np.ndarray, t_ctx: int, budget: int, n_sink: int, n_recent: int):
    """Score of the last middle position admitted at token level (the B-th boundary).

    Returns None when nothing is ranked (budget >= t_ctx or no free slot).
    """
    free = budget - n_sink - n_recent
    if budget >= t_ctx or free <= 0:
        return None
    mid = np.sort(score_row[n_sink: t_ctx - n_recent])[::-1]
    return float(mid[free - 1])


# ---------------------------------------------------------------------------
# One speculative step (Algorithm 2: sparsify, Draft x gamma, Verify).
# ---------------------------------------------------------------------------

def spec_step(k_cache, v_cache, q_win, q_draft, q_verify, t_ctx, budget, n_sink, n_recent,
              lse_win=None, chunk=1):
    """q_draft: [gamma, b, h_q, d]; q_verify: [b, h_q, gamma + 1, d].

    Returns a dict with idx, count, score, draft_o [gamma, b, h_q, d],
    draft_lse [gamma, b, h_q], verify_o, verify_lse.
    """
    idx, count, score = select_budget(q_win, k_cache, t_ctx, budget, n_sink, n_recent,
                                      chunk, lse_win)
    gamma = q_draft.shape[0]
    dos, dls = [], []
    for j in range(gamma):
        o, l = draft_attn(q_draft[j], k_cache, v_cache, idx, count, t_ctx, j)
        dos.append(o)
        dls.append(l)
    vo, vl = verify_attn(q_verify, k_cache, v_cache, t_ctx)
    return dict(idx=idx, count=count, score=score, draft_o=np.stack(dos),
                draft_lse=np.stack(dls), verify_o=vo, verify_lse=vl)


# ---------------------------------------------------------------------------
# Greedy acceptance (Eq. accept; Algorithm 2: longest matching prefix, then one
# verifier token).
# ---------------------------------------------------------------------------

def greedy_argmax(logits: np.ndarray) -> np.ndarray:
    """Token ids of the largest logit of every row (the arg max of Eq. accept).

    logits: [rows, vocab], compared in their own type.  Reading: ties go to the lowest
    token id, NaN logits are never chosen (-0 and +0 compare equal), and a row with no
    comparable logit gives id 0.
    """
    logits = np.asarray(logits)
    rows = logits.shape[0]
    out = np.zeros(rows, dtype=np.int64)
    for r in range(rows):
        row = logits[r]
        comparable = ~np.isnan(row)
        if comparable.any():
            top = row[comparable].max()
            out[r] = int(np.flatnonzero(row == top)[0])      # NaN == top is false
    return out


def accept_greedy(draft_tokens: np.ndarray, verify_tokens: np.ndarray):
    """Accepted length and emitted tokens of one verification (Algorithm 2).

    draft_tokens: [b, gamma] drafter tokens x_hat; verify_tokens: [b, gamma + 1]
    verifier tokens x_star at the same positions plus one past the block.  k is the
    largest count with x_hat[i] == x_star[i] for every i < k; the step emits
    x_hat[0:k] and then x_star[k].  Returns (k [b], emit [b, gamma + 1] padded
    with -1).
    """
    draft_tokens = np.asarray(draft_tokens)
    verify_tokens = np.asarray(verify_tokens)
    b, gamma = draft_tokens.shape
    n = np.zeros(b, dtype=np.int64)
    emit = np.full((b, gamma + 1), -1, dtype=np.int64)
    for bi in range(b):
        k = 0
        while k < gamma and draft_tokens[bi, k] == verify_tokens[bi, k]:
            k += 1
        n[bi] = k
        emit[bi, :k] = draft_tokens[bi, :k]
        emit[bi, k] = verify_tokens[bi, k]
    return n, emit


# ---------------------------------------------------------------------------
# Cache update after acceptance (Algorithm 2, Update): the accepted block rows join
# the context, the observation window slides over them, and the drafter's sparse
# view takes the accepted positions.
# ---------------------------------------------------------------------------

def batch_advance(n_accept: np.ndarray, n_q: int) -> int:
    """Positions every sequence of a batch that shares one context length advances by.

    Reading (the paper treats one sequence): sequence b keeps its block rows
    t_ctx .. t_ctx + n_accept[b] (the rows whose tokens are now settled: the token the
    block started from and the accepted drafts); a batch stored with one common length
    advances by the smallest of these counts, so every sequence stays on tokens its
    verifier has confirmed.
    """
    k = int(np.min(np.asarray(n_accept))) if np.asarray(n_accept).size else 0
    return min(max(k, 0), n_q - 1) + 1


def advance_window(q_win: np.ndarray, lse_win: np.ndarray, q_verify: np.ndarray,
                   lse_verify: np.ndarray, advance: int):
    """Slides the observation window by `advance` positions over the verified block.

    q_win [b, h_q, W, d] and lse_win [b, h_q, W] hold the queries and softmax
    normalisers of positions t_ctx - W .. t_ctx - 1; q_verify [b, h_q, n_q, d] and
    lse_verify [b, h_q, n_q] those of the block positions t_ctx .. t_ctx + n_q - 1.
    Returns the same arrays for positions t_ctx + advance - W .. t_ctx + advance - 1.
    """
    W = q_win.shape[2]
    q_all = np.concatenate([q_win, q_verify[:, :, :advance]], axis=2)
    l_all = np.concatenate([lse_win, lse_verify[:, :, :advance]], axis=2)
    return q_all[:, :, advance: advance + W].copy(), l_all[:, :, advance: advance + W].copy()


def append_view(idx: np.ndarray, count: np.ndarray, t_ctx: int, advance: int, capacity: int):
    """The sparse view after the settled block rows t_ctx .. t_ctx + advance - 1 join it.

    idx [b, h_kv, capacity] (ascending positions, -1 padding), count [b, h_kv].
    Returns new (idx, count); a view without room for the new rows is returned
    unchanged and flagged in the third result.
    """
    idx = np.array(idx, copy=True)
    count = np.array(count, copy=True)
    full = False
    for b in range(idx.shape[0]):
        for g in range(idx.shape[1]):
            c = int(count[b, g])
            if c + advance > capacity:
                full = True
                continue
            idx[b, g, c: c + advance] = np.arange(t_ctx, t_ctx + advance)
            count[b, g] = c + advance
    return idx, count, full


def widen_bf16_bits(bits: np.ndarray) -> np.ndarray:
    """Exact float64 value of bf16 bit patterns (uint16)."""
    bits = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return bits.view(np.float32).astype(np.float64)
