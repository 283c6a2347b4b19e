"""Ties under the paper's chunk policy (Sec. 3.4: the top floor(B/s) chunks, s = 8; ties go to
the lower chunk).  Middle keys set to zero give every middle position the same score, so every
full chunk has the same sum and the budget boundary falls among hundreds of tied chunks: the
chunk-level top-B must rank them exactly and keep the lowest."""

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W
from tests.parity import check_selection, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def test_tied_chunks_keep_the_lowest():
    wl = W.tiny_workload(batch=1, h_q=8, h_kv=2, head_dim=128, t_ctx=6000, budget=300, n_sink=4, n_recent=32,
                         window=32, gamma=1)
    inp = W.make_layer(wl, 0, "cuda")
    t, s = wl.t_ctx, 8
    lo, hi = wl.n_sink, t - wl.n_recent
    inp.k_cache[:, :, lo:hi].zero_()
    K, QW = f64(inp.k_cache), f64(inp.q_win)
    lse_ref = oracle.window_lse(QW, K, t)
    score_ref = oracle.window_scores(QW, K, lse_ref, t)
    idx_ref = np.full((wl.batch, wl.h_kv, wl.budget), -1)
    cnt_ref = np.zeros((wl.batch, wl.h_kv), dtype=np.int64)
    for b in range(wl.batch):
        for kv in range(wl.h_kv):
            keep = oracle.select_from_scores(score_ref[b, kv], t, wl.budget, wl.n_sink, wl.n_recent, s)
            idx_ref[b, kv, :keep.size] = keep
            cnt_ref[b, kv] = keep.size
    st = bd.SpecStep.for_workload(wl, chunk=s)
    st.select(inp.k_cache, inp.q_win, torch.from_numpy(lse_ref).float().cuda())
    torch.cuda.synchronize()
    check_selection(st.idx, st.count, idx_ref, cnt_ref, score_ref, t, wl.budget, wl.n_sink, wl.n_recent, s,
                    what="tied chunks")
    # exactly: chunk 0 holds the middle's first four positions only (a smaller sum), so the
    # kept chunks are 1 .. k, positions 8 .. 8 + 8k - 1, on both sides
    k = (wl.budget - wl.n_sink - wl.n_recent) // s
    want = np.concatenate([np.arange(lo), np.arange(s, s + s * k), np.arange(hi, t)])
    for b in range(wl.batch):
        for kv in range(wl.h_kv):
            assert np.array_equal(idx_ref[b, kv, : cnt_ref[b, kv]], want)
            kept = st.idx[b, kv, : int(st.count[b, kv])].cpu().numpy()
            assert np.array_equal(kept, want), (b, kv, kept[:12])
