"""Comparison helpers for the CUDA path against the fp64 oracle.

Tolerances:
  * attention outputs (bf16 inputs, fp32 accumulation, bf16 output):
      max-abs   max |o_gpu - o_ref|                                   <= 1e-2
      elem-rel  max |o_gpu - o_ref| / max(|o_ref|, 1e-3), element-wise <= 1e-2
      row-rel   max over rows of max_d |o_gpu - o_ref| / max_d |o_ref| <= 1e-2
                (implied by elem-rel; reported beside it)
      lse       max |lse_gpu - lse_ref|                               <= 1e-3
    Every check's figures are collected in RECORDS and printed at the end of the run.
  * selection: the kept sets have the same size and agree exactly, except for
    positions (chunks) whose oracle score lies within 1e-5 of the oracle's boundary
    score (the score of the last admitted middle position or chunk).
"""

from __future__ import annotations

import numpy as np
import torch

import oracle

ATOL = 1e-2
RTOL = 1e-2
LSE_ATOL = 1e-3
TIE_BAND = 1e-5
ELEM_FLOOR = 1e-3

RECORDS = []          # (what, figures) of every attention check of the session


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to(torch.float64).cpu().numpy()


def check_attention(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    o = f64(o_gpu)
    d = o.shape[-1]
    o = o.reshape(-1, d)
    r = np.asarray(o_ref, dtype=np.float64).reshape(-1, d)
    assert np.isfinite(o).all(), f"{what}: non-finite output"
    err = np.abs(o - r)
    max_abs = float(err.max()) if err.size else 0.0
    row_scale = np.maximum(np.abs(r).max(axis=1), 1e-6)
    max_rel = float((err.max(axis=1) / row_scale).max()) if err.size else 0.0
    elem_rel = float((err / np.maximum(np.abs(r), ELEM_FLOOR)).max()) if err.size else 0.0
    out = dict(max_abs=max_abs, elem_rel=elem_rel, max_rel=max_rel)
    RECORDS.append((what, out))
    assert max_abs <= ATOL, f"{what}: max-abs {max_abs:.3e} > {ATOL}"
    assert elem_rel <= RTOL, f"{what}: element-wise rel {elem_rel:.3e} > {RTOL}"
    assert max_rel <= RTOL, f"{what}: max-rel {max_rel:.3e} > {RTOL}"
    if lse_gpu is not None:
        lg = f64(lse_gpu).reshape(-1)
        lr = np.asarray(lse_ref, dtype=np.float64).reshape(-1)
        both_inf = np.isneginf(lg) & np.isneginf(lr)
        assert np.array_equal(np.isneginf(lg), np.isneginf(lr)), f"{what}: -inf lse mismatch"
        lerr = np.zeros_like(lg)
        lerr[~both_inf] = np.abs(lg[~both_inf] - lr[~both_inf])
        assert lerr.max() <= LSE_ATOL, f"{what}: lse err {lerr.max():.3e}"
        out["lse_abs"] = float(lerr.max())
    return out


def chunk_scores(score_row, t_ctx, n_sink, n_recent, chunk):
    lo, hi = n_sink, t_ctx - n_recent
    first, last = lo // chunk, (hi - 1) // chunk
    ids = np.arange(first, last + 1)
    vals = np.array([score_row[max(c * chunk, lo): min(c * chunk + chunk, hi)].sum() for c in ids])
    return ids, vals


def check_selection(idx_gpu, count_gpu, idx_ref, count_ref, score_ref, t_ctx, budget, n_sink, n_recent,
                    chunk=1, what=""):
    """Returns the number of positions that differ (all inside the tie band)."""
    idx = idx_gpu.cpu().numpy().reshape(-1, budget)
    cnt = count_gpu.cpu().numpy().reshape(-1)
    iref = np.asarray(idx_ref).reshape(-1, budget)
    cref = np.asarray(count_ref).reshape(-1)
    sref = np.asarray(score_ref).reshape(iref.shape[0], -1)
    assert np.array_equal(cnt, cref), f"{what}: counts {cnt[:8]} vs {cref[:8]}"
    n_diff = 0
    for u in range(idx.shape[0]):
        g = idx[u, : cnt[u]]
        r = iref[u, : cref[u]]
        assert np.all((g >= 0) & (g < t_ctx)), f"{what}: unit {u} out-of-range position"
        assert np.all(np.diff(g) > 0), f"{what}: unit {u} not ascending/unique"
        assert np.all(idx[u, cnt[u]:] == -1), f"{what}: unit {u} padding"
        if budget < t_ctx:
            assert set(range(n_sink)) <= set(g.tolist()), f"{what}: unit {u} lost a sink"
            assert set(range(t_ctx - n_recent, t_ctx)) <= set(g.tolist()), f"{what}: unit {u} lost a recent"
        diff = np.setxor1d(g, r)
        if diff.size == 0:
            continue
        n_diff += diff.size
        if chunk == 1:
            tau = oracle.boundary_score(sref[u], t_ctx, budget, n_sink, n_recent)
            assert tau is not None, f"{what}: unit {u} differs without a ranking"
            gap = np.abs(sref[u][diff] - tau)
            assert gap.max() <= TIE_BAND, f"{what}: unit {u} positions {diff[:6]} differ, gap {gap.max():.3e}"
        else:
            ids, vals = chunk_scores(sref[u], t_ctx, n_sink, n_recent, chunk)
            k = (budget - n_sink - n_recent) // chunk
            tau = np.sort(vals)[::-1][k - 1]
            cdiff = np.unique(diff // chunk)
            gap = np.abs(vals[np.searchsorted(ids, cdiff)] - tau)
            assert gap.max() <= TIE_BAND, f"{what}: unit {u} chunks {cdiff[:6]} differ, gap {gap.max():.3e}"
    return n_diff
