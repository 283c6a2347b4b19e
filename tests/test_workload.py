"""The seeded input recipe (CPU): the five workloads' shapes, reproducible draws, per-sequence
draws that match the batched ones (the host-core baseline draws sequence by sequence), and
the planted heavy hitters."""

import dataclasses

import numpy as np
import torch

from paper_2606_00144_gb300 import workload as W


def test_the_five_workloads():
    # batch, h_q, h_kv, d, T, B, sink, recent, layers, heavy-hitter fraction (or range)
    want = {
        "tiny_1k": (1, 8, 2, 64, 1024, 256, 4, 64, 1, 0.02),
        "l8b_4k": (1, 32, 8, 128, 4096, 512, 4, 128, 1, 0.02),
        "l8b_8k_b4": (4, 32, 8, 128, 8192, 1024, 4, 256, 1, 0.01),
        "l8b_16k_b8": (8, 32, 8, 128, 16384, 512, 4, 128, 1, 0.01),
        "l8b_32L_16k_b16": (16, 32, 8, 128, 16384, 512, 4, 128, 32, (0.005, 0.03)),
    }
    assert set(W.WORKLOADS) == set(want)
    for name, (b, hq, hkv, d, t, budget, sink, recent, layers, hh) in want.items():
        wl = W.WORKLOADS[name]
        assert (wl.batch, wl.h_q, wl.h_kv, wl.head_dim, wl.t_ctx, wl.budget, wl.n_sink, wl.n_recent,
                wl.layers) == (b, hq, hkv, d, t, budget, sink, recent, layers), name
        assert (wl.hh_frac_range if isinstance(hh, tuple) else wl.hh_frac) == hh, name
        assert wl.window == 32 and wl.gamma == 5 and wl.t_cap == t + 6
        # the middle's free slots: B - S - R (188 / 380 / 764 / 380 / 380)
        assert budget - sink - recent == {1024: 188, 4096: 380, 8192: 764}.get(t, 380)
    assert W.SWEEP_16K == (256, 512, 1024, 2048, 16384)


def test_budget_sweep_keeps_a_quarter_recent():
    wl = W.WORKLOADS["l8b_16k_b8"].with_budget(2048)
    assert (wl.budget, wl.n_recent, wl.n_sink) == (2048, 512, 4)


def test_draws_are_reproducible_and_bf16():
    wl = W.tiny_workload(batch=2, h_q=4, h_kv=2, head_dim=64, t_ctx=300, gamma=3)
    a, b = W.make_layer(wl, 0), W.make_layer(wl, 0)
    for name in ("k_cache", "v_cache", "q_win", "q_draft", "q_verify"):
        x, y = getattr(a, name), getattr(b, name)
        assert x.dtype == torch.bfloat16 and torch.equal(x, y), name
    assert a.k_cache.shape == (2, 2, 300 + 4, 64)
    assert a.q_win.shape == (2, 4, 32, 64) and a.q_draft.shape == (3, 2, 4, 64)
    assert a.q_verify.shape == (2, 4, 4, 64)
    c = W.make_layer(wl, 1)
    assert not torch.equal(a.k_cache, c.k_cache), "layers must draw different inputs"
    assert not torch.equal(a.k_cache[0], a.k_cache[1]), "sequences must draw different inputs"


def test_one_sequence_at_a_time_matches_the_batch():
    wl = W.tiny_workload(batch=3, h_q=4, h_kv=2, head_dim=64, t_ctx=250, gamma=2)
    full = W.make_layer(wl, 2)
    one = dataclasses.replace(wl, batch=1)
    for bi in range(wl.batch):
        s = W.make_layer(one, 2, first_seq=bi)
        assert torch.equal(s.k_cache[0], full.k_cache[bi])
        assert torch.equal(s.v_cache[0], full.v_cache[bi])
        assert torch.equal(s.q_win[0], full.q_win[bi])
        assert torch.equal(s.q_draft[:, 0], full.q_draft[:, bi])
        assert torch.equal(s.q_verify[0], full.q_verify[bi])


def test_heavy_hitters_are_planted_along_the_group_query_direction():
    wl = W.tiny_workload(batch=2, h_q=8, h_kv=2, head_dim=128, t_ctx=4000, gamma=1, hh_frac=0.02)
    inp = W.make_layer(wl, 0)
    n_hh = int(0.02 * 4000)
    k = inp.k_cache.float()
    for bi in range(wl.batch):
        for kv in range(wl.h_kv):
            pos = inp.hh_pos[bi * wl.h_kv + kv].numpy()
            assert pos.size == n_hh and np.unique(pos).size == n_hh
            assert pos.min() >= 0 and pos.max() < wl.t_ctx
            qsum = inp.q_win[bi, kv * wl.group:(kv + 1) * wl.group].float().sum(dim=(0, 1))
            u = qsum / qsum.norm()
            proj = (k[bi, kv, : wl.t_ctx] @ u).numpy()
            rest = np.setdiff1d(np.arange(wl.t_ctx), pos)
            # planted keys carry +3 along u (bf16 rounding aside); the others are N(0, 1) there
            assert abs(proj[pos].mean() - 3.0) < 0.35, proj[pos].mean()
            assert abs(proj[rest].mean()) < 0.1 and 0.8 < proj[rest].std() < 1.2


def test_stack_fraction_is_drawn_per_layer_in_range():
    wl = W.WORKLOADS["l8b_32L_16k_b16"]
    fr = [W.layer_hh_frac(wl, l) for l in range(wl.layers)]
    assert all(0.005 <= f <= 0.03 for f in fr)
    assert len(set(fr)) == wl.layers
    assert fr == [W.layer_hh_frac(wl, l) for l in range(wl.layers)]
