"""Parity of the CUDA path (through the C ABI) with the fp64 oracle on the same seeded inputs.

Covers the five evaluation workloads (the 32-layer stack on whole and sampled layers), the
16K budget sweep including the B >= T case, ragged shapes that span several tiles with a
partial tail, the degenerate cases, the standalone merge and determinism.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W
from tests.parity import check_attention, check_selection, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="session", autouse=True)
def built():
    bd.build()
    bd.library()


def host(inp):
    return dict(K=f64(inp.k_cache), V=f64(inp.v_cache), QW=f64(inp.q_win), QD=f64(inp.q_draft),
                QV=f64(inp.q_verify))


def run_and_check(wl, inp, h, budgets=None, modes=("carry", "self"), chunk=1, check_steps=True, tag="",
                  recent=None):
    """Runs selection (both modes), gamma drafts on the oracle's selection, and verify.
    recent: the recent window of every budget (default: the workload's for its own budget,
    budget // 4 for the others)."""
    t = wl.t_ctx
    lse_ref = oracle.window_lse(h["QW"], h["K"], t)
    score_ref = oracle.window_scores(h["QW"], h["K"], lse_ref, t)
    lse_dev = torch.from_numpy(lse_ref).float().cuda()
    stats = {}
    budgets = budgets or [wl.budget]
    for budget in budgets:
        n_recent = recent if recent is not None else (wl.n_recent if budget == wl.budget else budget // 4)
        st = bd.SpecStep.for_workload(wl, budget=budget, n_recent=n_recent, chunk=chunk)
        idx_ref = np.full((wl.batch, wl.h_kv, budget), -1)
        cnt_ref = np.zeros((wl.batch, wl.h_kv), dtype=np.int64)
        for b in range(wl.batch):
            for kv in range(wl.h_kv):
                keep = oracle.select_from_scores(score_ref[b, kv], t, budget, wl.n_sink, n_recent, chunk)
                idx_ref[b, kv, : keep.size] = keep
                cnt_ref[b, kv] = keep.size
        for mode in modes:
            # both orders of the window-query load: early (BD_SELECT_WINDOW_READY) in carry
            # mode, after the dependency wait in self mode
            st.select(inp.k_cache, inp.q_win, lse_dev if mode == "carry" else None, window_ready=mode == "carry")
            torch.cuda.synchronize()
            nd = check_selection(st.idx, st.count, idx_ref, cnt_ref, score_ref, t, budget, wl.n_sink, n_recent,
                                 chunk, what=f"{tag} B={budget} {mode}")
            stats[f"select_B{budget}_{mode}_diff"] = nd
        if not check_steps:
            continue
        # drafts on the oracle's selection (both sides see the same sparse view)
        st.idx.copy_(torch.from_numpy(idx_ref).int())
        st.count.copy_(torch.from_numpy(cnt_ref).int())
        for j in range(wl.gamma):
            # passes after the first gather the view before the previous pass has finished
            st.draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache, view_ready=j > 0)
            o_ref, l_ref = oracle.draft_attn(h["QD"][j], h["K"], h["V"], idx_ref, cnt_ref, t, j)
            torch.cuda.synchronize()
            stats[f"draft{j}_B{budget}"] = check_attention(st.draft_o[j], st.draft_lse[j], o_ref, l_ref,
                                                           f"{tag} draft j={j} B={budget}")
        if budget == budgets[0]:
            st.verify(inp.q_verify, inp.k_cache, inp.v_cache)
            o_ref, l_ref = oracle.verify_attn(h["QV"], h["K"], h["V"], t)
            torch.cuda.synchronize()
            stats["verify"] = check_attention(st.verify_o, st.verify_lse, o_ref, l_ref, f"{tag} verify")
        assert st.ws.status() == 0
    return stats


# ----------------------------------------------------------------------------- evaluation workloads

def test_tiny_1k():
    wl = W.WORKLOADS["tiny_1k"]
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), tag="tiny_1k")


def test_l8b_4k():
    wl = W.WORKLOADS["l8b_4k"]
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), tag="l8b_4k")


def test_l8b_8k_b4():
    wl = W.WORKLOADS["l8b_8k_b4"]
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), tag="l8b_8k_b4")


def test_l8b_16k_b8_budget_sweep():
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), budgets=list(W.SWEEP_16K), modes=("carry",), tag="l8b_16k_b8")


def test_l8b_16k_b8_chunk_policy():
    """The paper's policy (Sec. 3.4): the top floor(B/8) chunks of 8 by cumulative attention
    with no sink or recent window, over the budget sweep; then s = 8 beside the default
    sink and recent window."""
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    h = host(inp)
    pure = dataclasses.replace(wl, n_sink=0, n_recent=0)
    run_and_check(pure, inp, h, budgets=[512, 256, 1024, 2048], chunk=8, recent=0, modes=("carry",),
                  tag="chunk8 pure")
    run_and_check(wl, inp, h, chunk=8, modes=("carry", "self"), check_steps=False, tag="chunk8")


def test_l8b_16k_b8_self_mode_selection():
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), modes=("self",), check_steps=False, tag="l8b_16k_b8")


def test_full_budget_draft_equals_full_attention():
    # B >= T: the sparse view is the whole prefix, so draft pass j equals full causal attention
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    st = bd.SpecStep.for_workload(wl, budget=16384, n_recent=4096)
    st.select(inp.k_cache, inp.q_win, None)
    torch.cuda.synchronize()
    assert (st.count == wl.t_ctx).all()
    assert torch.equal(st.idx[..., : wl.t_ctx].cpu(), torch.arange(wl.t_ctx).expand(wl.batch, wl.h_kv, -1).int())
    K, V = f64(inp.k_cache), f64(inp.v_cache)
    for j in (0, wl.gamma - 1):
        st.draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache)
        q_blk = np.zeros((wl.batch, wl.h_q, j + 1, wl.head_dim))
        q_blk[:, :, j] = f64(inp.q_draft[j])
        o_ref, l_ref = oracle.verify_attn(q_blk, K, V, wl.t_ctx)
        torch.cuda.synchronize()
        check_attention(st.draft_o[j], st.draft_lse[j], o_ref[:, :, j], l_ref[:, :, j], f"full-budget draft {j}")


def _unit_slice(inp, b, kv, group):
    hs = slice(kv * group, (kv + 1) * group)
    return dict(K=f64(inp.k_cache[b:b + 1, kv:kv + 1]), V=f64(inp.v_cache[b:b + 1, kv:kv + 1]),
                QW=f64(inp.q_win[b:b + 1, hs]), QD=f64(inp.q_draft[:, b:b + 1, hs]),
                QV=f64(inp.q_verify[b:b + 1, hs]))


@pytest.mark.slow
@pytest.mark.parametrize("layer,units", [(0, "all"), (31, [(0, 0), (7, 3), (15, 7)])])
def test_l8b_32L_16k_b16_layers(layer, units):
    wl = W.WORKLOADS["l8b_32L_16k_b16"]
    inp = W.make_layer(wl, layer, "cuda")
    st = bd.SpecStep.for_workload(wl)
    lse_dev = st.window_lse(inp.k_cache, inp.q_win)     # carry state as a previous verify leaves it
    st.run(inp.k_cache, inp.v_cache, inp.q_win, inp.q_draft, inp.q_verify, window_lse=lse_dev)
    torch.cuda.synchronize()
    if units == "all":
        units = [(b, kv) for b in range(wl.batch) for kv in range(wl.h_kv)]
    g, t = wl.group, wl.t_ctx
    for b, kv in units:
        h = _unit_slice(inp, b, kv, g)
        lse_ref = oracle.window_lse(h["QW"], h["K"], t)
        lse_gpu = f64(lse_dev[b, kv * g:(kv + 1) * g]).reshape(-1)
        assert np.abs(lse_gpu - lse_ref.reshape(-1)).max() <= 1e-3
        score = oracle.window_scores(h["QW"], h["K"], lse_ref, t)
        keep = oracle.select_from_scores(score[0, 0], t, wl.budget, wl.n_sink, wl.n_recent)
        idx_ref = np.full((1, 1, wl.budget), -1)
        idx_ref[0, 0, : keep.size] = keep
        check_selection(st.idx[b, kv], st.count[b, kv], idx_ref, np.array([keep.size]), score, t, wl.budget,
                        wl.n_sink, wl.n_recent, what=f"32L layer {layer} ({b},{kv})")
        vo, vl = oracle.verify_attn(h["QV"], h["K"], h["V"], t)
        check_attention(st.verify_o[b, kv * g:(kv + 1) * g], st.verify_lse[b, kv * g:(kv + 1) * g], vo, vl,
                        f"32L verify ({b},{kv})")
        # drafts ran on the GPU's selection; compare where it equals the oracle's (else ties decided it)
        gsel = st.idx[b, kv, : int(st.count[b, kv])].cpu().numpy()
        if np.array_equal(gsel, keep):
            for j in (0, wl.gamma - 1):
                do, dl = oracle.draft_attn(h["QD"][j], h["K"], h["V"], idx_ref, np.array([[keep.size]]), t, j)
                check_attention(st.draft_o[j, b, kv * g:(kv + 1) * g], st.draft_lse[j, b, kv * g:(kv + 1) * g],
                                do, dl, f"32L draft {j} ({b},{kv})")
    assert st.ws.status() == 0


# ----------------------------------------------------------------------------- ragged and degenerate shapes

RAGGED = [
    # batch, h_q, h_kv, d, t_ctx, budget, sink, recent, window, gamma, chunk
    (2, 8, 2, 128, 777, 100, 4, 20, 32, 5, 1),
    (1, 4, 4, 64, 65, 16, 1, 3, 8, 3, 1),         # group 1, d 64, tail of one key
    (3, 16, 2, 64, 333, 64, 0, 0, 16, 2, 1),      # group 8, no sink/recent
    (1, 4, 1, 128, 1000, 200, 4, 8, 32, 5, 1),    # window wider than the recent set: causal scores
    (2, 8, 2, 128, 640, 136, 0, 0, 32, 5, 8),     # the paper's chunk policy, s = 8
    (1, 8, 2, 128, 1031, 128, 4, 32, 32, 5, 8),   # chunks with sink/recent and ragged chunk edges
    (1, 8, 2, 128, 300, 36, 4, 32, 32, 1, 1),     # B = sink + recent: nothing ranked
    (1, 8, 2, 64, 40, 64, 4, 8, 32, 5, 1),        # B > T
    (1, 16, 2, 128, 700, 100, 4, 16, 32, 2, 1),   # group 8 x window 32 = 256 rows: two TMEM accumulators, one Q buffer
    (2, 16, 2, 64, 900, 120, 4, 16, 32, 2, 1),    # the same at d 64
    (1, 8, 2, 128, 20000, 600, 4, 64, 32, 1, 1),  # 16K < middle <= 32K: the shared-memory top-B kernel
    (1, 4, 1, 64, 40000, 300, 4, 32, 32, 1, 1),   # middle > 32K: the general top-B kernel
]


@pytest.mark.parametrize("case", RAGGED)
def test_ragged_shapes(case):
    b, hq, hkv, d, t, budget, sink, recent, window, gamma, chunk = case
    wl = W.tiny_workload(batch=b, h_q=hq, h_kv=hkv, head_dim=d, t_ctx=t, budget=budget, n_sink=sink,
                         n_recent=recent, window=window, gamma=gamma, seed=11 + t)
    inp = W.make_layer(wl, 0, "cuda")
    modes = ("carry", "self") if (hq // hkv) * window <= 128 else ("carry",)   # self mode: <= 128 window rows
    run_and_check(wl, inp, host(inp), chunk=chunk, tag=f"ragged{case}", modes=modes)


@pytest.mark.parametrize("n_q,with_v", [(1, True), (2, True), (12, True), (21, True), (32, False)])
def test_verify_block_sizes(n_q, with_v):
    wl = W.tiny_workload(batch=2, h_q=8, h_kv=2, head_dim=128, t_ctx=1500, gamma=n_q - 1 if n_q > 1 else 1)
    inp = W.make_layer(wl, 0, "cuda")
    g = torch.Generator(device="cuda").manual_seed(900 + n_q)
    q = torch.randn(wl.batch, wl.h_q, n_q, wl.head_dim, device="cuda", generator=g).to(torch.bfloat16)
    shape = bd.shape_of(inp.k_cache, wl.h_q, wl.t_ctx)
    ws = bd.Workspace(bd.bd_workspace_size(shape, bd.BD_OP_VERIFY, 1, n_q))
    o = torch.empty(wl.batch, wl.h_q, n_q, wl.head_dim, dtype=torch.bfloat16, device="cuda") if with_v else None
    lse = torch.empty(wl.batch, wl.h_q, n_q, device="cuda")
    bd.bd_verify_attn(shape, q, n_q, inp.k_cache, inp.v_cache, o, lse, ws)
    o_ref, l_ref = oracle.verify_attn(f64(q), f64(inp.k_cache), f64(inp.v_cache), wl.t_ctx)
    torch.cuda.synchronize()
    if with_v:
        check_attention(o, lse, o_ref, l_ref, f"verify n_q={n_q}")
    else:
        assert np.abs(f64(lse) - l_ref).max() <= 1e-3


@pytest.mark.parametrize("h_q,h_kv,d,t_ctx,n_q", [(32, 4, 128, 1500, 21), (32, 4, 64, 777, 13), (32, 2, 128, 900, 21),
                                                   (32, 4, 128, 16384, 21)])
def test_verify_blocks_beyond_one_cta(h_q, h_kv, d, t_ctx, n_q):
    """More query rows per KV head than one CTA's warps hold (96): G = 8 with the paper's
    gamma = 20 (168 rows, two chunks), 104 rows, and G = 16 (336 rows, four chunks), the last
    case at 16K context."""
    wl = W.tiny_workload(batch=2, h_q=h_q, h_kv=h_kv, head_dim=d, t_ctx=t_ctx, gamma=n_q - 1)
    inp = W.make_layer(wl, 0, "cuda")
    g = torch.Generator(device="cuda").manual_seed(4242 + n_q)
    q = torch.randn(wl.batch, wl.h_q, n_q, d, device="cuda", generator=g).to(torch.bfloat16)
    shape = bd.shape_of(inp.k_cache, wl.h_q, wl.t_ctx)
    ws = bd.Workspace(bd.bd_workspace_size(shape, bd.BD_OP_VERIFY, 1, n_q))
    o = torch.empty(wl.batch, wl.h_q, n_q, d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(wl.batch, wl.h_q, n_q, device="cuda")
    for rep in range(2):                       # the workspace is reused as in a loop of steps
        o.fill_(7)
        bd.bd_verify_attn(shape, q, n_q, inp.k_cache, inp.v_cache, o, lse, ws)
        torch.cuda.synchronize()
        o_ref, l_ref = oracle.verify_attn(f64(q), f64(inp.k_cache), f64(inp.v_cache), wl.t_ctx)
        check_attention(o, lse, o_ref, l_ref, f"verify G={h_q // h_kv} n_q={n_q} T={t_ctx} rep {rep}")
    assert ws.status() == 0


def test_verify_chunked_block_with_per_sequence_lengths():
    lens = [1500, 977, 64]
    b, h_q, h_kv, d, n_q = len(lens), 32, 4, 128, 21
    wl = W.tiny_workload(batch=b, h_q=h_q, h_kv=h_kv, head_dim=d, t_ctx=max(lens), gamma=n_q - 1)
    inp = W.make_layer(wl, 0, "cuda")
    g = torch.Generator(device="cuda").manual_seed(77)
    q = torch.randn(b, h_q, n_q, d, device="cuda", generator=g).to(torch.bfloat16)
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    shape = bd.make_shape(b, h_q, h_kv, d, max(lens), wl.t_cap, seq_lens=lens_d)
    ws = bd.Workspace(bd.bd_workspace_size(shape, bd.BD_OP_VERIFY, 1, n_q))
    o = torch.empty(b, h_q, n_q, d, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(b, h_q, n_q, device="cuda")
    bd.bd_verify_attn(shape, q, n_q, inp.k_cache, inp.v_cache, o, lse, ws)
    torch.cuda.synchronize()
    K, V, Q = f64(inp.k_cache), f64(inp.v_cache), f64(q)
    for i, t in enumerate(lens):
        o_ref, l_ref = oracle.verify_attn(Q[i:i + 1], K[i:i + 1], V[i:i + 1], t)
        check_attention(o[i:i + 1], lse[i:i + 1], o_ref, l_ref, f"chunked verify seq {i} T={t}")
    assert ws.status() == 0


def test_draft_empty_view_and_full_view():
    wl = W.tiny_workload(batch=2, h_q=8, h_kv=2, head_dim=128, t_ctx=500, budget=64)
    inp = W.make_layer(wl, 0, "cuda")
    h = host(inp)
    st = bd.SpecStep.for_workload(wl)
    rng = np.random.default_rng(3)
    idx = np.full((2, 2, 64), -1)
    cnt = np.array([[0, 64], [17, 1]])
    for b in range(2):
        for kv in range(2):
            idx[b, kv, : cnt[b, kv]] = np.sort(rng.choice(500, cnt[b, kv], replace=False))
    st.idx.copy_(torch.from_numpy(idx).int())
    st.count.copy_(torch.from_numpy(cnt).int())
    for j in range(wl.gamma):
        st.draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache)
        o_ref, l_ref = oracle.draft_attn(h["QD"][j], h["K"], h["V"], idx, cnt, wl.t_ctx, j)
        torch.cuda.synchronize()
        check_attention(st.draft_o[j], st.draft_lse[j], o_ref, l_ref, f"draft edge j={j}")


def test_draft_out_of_range_index_is_reported_and_masked():
    wl = W.tiny_workload(batch=1, h_q=4, h_kv=1, head_dim=64, t_ctx=100, budget=8)
    inp = W.make_layer(wl, 0, "cuda")
    h = host(inp)
    st = bd.SpecStep.for_workload(wl)
    idx = np.array([[[0, 5, 9, 100000, 20, -1, -1, -1]]])
    st.idx.copy_(torch.from_numpy(idx).int())
    st.count.fill_(5)
    st.draft(0, inp.q_draft[0], inp.k_cache, inp.v_cache)
    torch.cuda.synchronize()
    assert st.ws.status() == -1                             # BD_ERR_INVALID_ARG recorded on the device
    good = np.array([[[0, 5, 9, 20]]])
    o_ref, l_ref = oracle.draft_attn(h["QD"][0], h["K"], h["V"], good, np.array([[4]]), wl.t_ctx, 0)
    check_attention(st.draft_o[0], st.draft_lse[0], o_ref, l_ref, "draft masked bad index")
    assert st.ws.status() == 0                              # reading clears it


def test_combine_standalone():
    rng = np.random.default_rng(5)
    for n_split, rows, d in [(1, 3, 64), (5, 37, 128), (40, 9, 128)]:
        o_part = rng.standard_normal((n_split, rows, d)).astype(np.float32)
        lse_part = (rng.standard_normal((n_split, rows)) * 3).astype(np.float32)
        lse_part[rng.random((n_split, rows)) < 0.2] = -np.inf
        lse_part[:, 0] = -np.inf                     # an all-empty row
        o_dev = torch.from_numpy(o_part).cuda()
        l_dev = torch.from_numpy(lse_part).cuda()
        out = torch.empty(rows, d, dtype=torch.bfloat16, device="cuda")
        lse = torch.empty(rows, device="cuda")
        bd.bd_combine(o_dev, l_dev, n_split, rows, d, out, lse)
        o_ref, l_ref = oracle.combine(o_part.astype(np.float64), lse_part.astype(np.float64))
        torch.cuda.synchronize()
        check_attention(out, lse, o_ref, l_ref, f"combine {n_split}x{rows}x{d}")


def test_combine_merges_disjoint_draft_views():
    """Draft attention over two disjoint halves of a view, merged by bd_combine, equals draft
    attention over the whole view.  The halves' results (the parts a split-K caller hands to
    bd_combine, in its fp32 input type) come from the oracle's draft pass; the GPU's own
    split-K drafts are checked in every draft parity case."""
    wl = W.tiny_workload(batch=1, h_q=8, h_kv=2, head_dim=128, t_ctx=900, budget=128)
    inp = W.make_layer(wl, 0, "cuda")
    h = host(inp)
    rng = np.random.default_rng(9)
    full = np.stack([np.sort(rng.choice(900, 128, replace=False)) for _ in range(2)])[None]
    parts_o, parts_l = [], []
    for half in (slice(0, 64), slice(64, 128)):
        sub = np.full((1, 2, 128), -1)
        sub[..., :64] = full[..., half]
        o, l = oracle.draft_attn(h["QD"][0], h["K"], h["V"], sub, np.full((1, 2), 64), 900, 0)
        parts_o.append(o.reshape(-1, 128))
        parts_l.append(l.reshape(-1))
    o_part = torch.from_numpy(np.stack(parts_o)).float().cuda()
    l_part = torch.from_numpy(np.stack(parts_l)).float().cuda()
    out = torch.empty(8, 128, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(8, device="cuda")
    bd.bd_combine(o_part, l_part, 2, 8, 128, out, lse)
    # each part also attended to the drafted row t_ctx: the union counts it twice
    both = np.concatenate([full[0], np.full((2, 2), 900)], axis=1)
    o_ref = np.zeros((8, 128))
    l_ref = np.zeros(8)
    for hh in range(8):
        kv = hh // 4
        o_ref[hh], l_ref[hh] = oracle.attention(h["QD"][0, 0, hh], h["K"][0, kv, both[kv]], h["V"][0, kv, both[kv]],
                                                1 / np.sqrt(128))
    torch.cuda.synchronize()
    check_attention(out, lse, o_ref, l_ref, "combine of draft parts")


@pytest.mark.parametrize("planted", [0, 100])
def test_tied_scores_take_lowest_positions(planted):
    """Middle keys set to zero have exactly equal scores: all of them (planted = 0: min = max)
    or all but every planted-th key, with the boundary falling among the ties in a bin too
    crowded to rank, so the exact radix select runs."""
    wl = W.tiny_workload(batch=1, h_q=8, h_kv=2, head_dim=128, t_ctx=6000, budget=300, n_sink=4, n_recent=32,
                         window=32, gamma=1)
    inp = W.make_layer(wl, 0, "cuda")
    mid = inp.k_cache[:, :, wl.n_sink: wl.t_ctx - wl.n_recent]
    keep = mid[:, :, ::planted].clone() if planted else None
    mid.zero_()
    if planted:
        mid[:, :, ::planted] = keep
    run_and_check(wl, inp, host(inp), check_steps=False, tag=f"ties planted={planted}")


def test_boundary_among_underflowed_scores():
    """Window queries along one axis and middle keys pointing the other way: their scores
    underflow to exactly 0 in fp32 (the oracle's fp64 values are ~1e-150, inside the tie
    band), only every 100th key scores above 0, so the budget boundary falls among the
    zeros.  The top-B then has to take real zero-score positions in position order ahead
    of the zero padding of its register rows (5964 middle scores in 8192 slots)."""
    wl = W.tiny_workload(batch=1, h_q=8, h_kv=2, head_dim=128, t_ctx=6000, budget=300, n_sink=4, n_recent=32,
                         window=32, gamma=1)
    inp = W.make_layer(wl, 0, "cuda")
    inp.q_win.mul_(0.05)
    inp.q_win[..., 0] = 64.0
    mid = inp.k_cache[:, :, wl.n_sink: wl.t_ctx - wl.n_recent]
    mid.mul_(0.05)
    mid[..., 0] = -64.0
    mid[:, :, ::100, 0] = 64.0
    run_and_check(wl, inp, host(inp), check_steps=False, tag="boundary among zero scores")


@pytest.mark.parametrize("run", [4, 64])
def test_exact_ties_ranked_above_the_bound(run):
    """Middle keys repeated in runs of `run` identical rows, so scores tie exactly in runs,
    and the top-B that ranks only the scores above the bound from group maxima meets its
    boundary inside a run (k = 266 is no multiple of 4): four ties in the boundary bin
    (ranked by one warp) or 64 (ranked by the whole CTA).  Besides the check against the
    oracle, the run that the boundary splits must keep its lowest positions (Sec. 3.4 top-k,
    ties to the lower index): identical keys have identical scores by definition."""
    wl = W.tiny_workload(batch=2, h_q=8, h_kv=2, head_dim=128, t_ctx=4096, budget=302, n_sink=4, n_recent=32,
                         window=32, gamma=1, seed=77 + run)
    inp = W.make_layer(wl, 0, "cuda")
    lo, hi = wl.n_sink, wl.t_ctx - wl.n_recent
    mid = inp.k_cache[:, :, lo:hi]
    first = torch.arange(hi - lo, device=mid.device) // run * run
    mid.copy_(mid[:, :, first].clone())
    h = host(inp)
    run_and_check(wl, inp, h, modes=("carry",), check_steps=False, tag=f"runs of {run}")
    t = wl.t_ctx
    lse_ref = oracle.window_lse(h["QW"], h["K"], t)
    st = bd.SpecStep.for_workload(wl)
    st.select(inp.k_cache, inp.q_win, torch.from_numpy(lse_ref).float().cuda())
    torch.cuda.synchronize()
    n_split = 0
    for b in range(wl.batch):
        for kv in range(wl.h_kv):
            kept = st.idx[b, kv, : int(st.count[b, kv])].cpu().numpy()
            kept = kept[(kept >= lo) & (kept < hi)] - lo
            taken = np.bincount(kept // run, minlength=(hi - lo + run - 1) // run)
            size = np.bincount(np.arange(hi - lo) // run)
            for r in np.nonzero((taken > 0) & (taken < size))[0]:
                assert np.array_equal(np.sort(kept[kept // run == r]), r * run + np.arange(taken[r])), \
                    f"unit ({b},{kv}) run {r}: kept {np.sort(kept[kept // run == r])[:8]} are not its lowest positions"
                n_split += 1
    assert n_split > 0, "no run was split by the boundary"


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("h_q", [18, 32])
def test_groups_beyond_one_query_tile(h_q, d):
    """GQA groups of 9 and 16 query heads per KV head: the draft kernel holds the group in two
    n8 query tiles (the selection with a 16-row window keeps G * W <= 256 rows; carry mode,
    as self mode takes at most 128 window rows), checked step by step against the oracle."""
    wl = W.tiny_workload(batch=2, h_q=h_q, h_kv=2, head_dim=d, t_ctx=900, budget=128, n_sink=4, n_recent=16,
                         window=16, gamma=3)
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), modes=("carry",), tag=f"group {h_q // 2} d{d}")


@pytest.mark.parametrize("d", [64, 128])
def test_self_mode_whole_units_per_cta(d):
    """128 (sequence, KV head) units of one 128-key tile each: every CTA of the window-LSE
    kernel holds whole units, so each unit's normalisers are written directly (no segment
    merge), next to the split-unit path the longer workloads take."""
    wl = W.tiny_workload(batch=16, h_q=32, h_kv=8, head_dim=d, t_ctx=120, budget=64, n_sink=4, n_recent=16,
                         window=32, gamma=2)
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), modes=("self",), check_steps=False, tag=f"whole units d{d}")


def test_determinism():
    wl = W.WORKLOADS["l8b_4k"]
    inp = W.make_layer(wl, 0, "cuda")
    outs = []
    for _ in range(2):
        st = bd.SpecStep.for_workload(wl)
        st.run(inp.k_cache, inp.v_cache, inp.q_win, inp.q_draft, inp.q_verify)
        torch.cuda.synchronize()
        outs.append([t.clone() for t in (st.idx, st.count, st.draft_o, st.draft_lse, st.verify_o, st.verify_lse)])
    for a, b in zip(*outs):
        assert torch.equal(a, b)


@pytest.mark.parametrize("group", [3, 5, 7])
def test_groups_not_a_power_of_two(group):
    """GQA groups of 3, 5 and 7 (Qwen-style 28/4): selection, every draft pass (the query
    tile holds the group's rows, the rest padding) and verify against the oracle."""
    wl = W.tiny_workload(batch=2, h_q=2 * group, h_kv=2, head_dim=128, t_ctx=900, budget=120, n_sink=4,
                         n_recent=16, window=16, gamma=3, seed=23 + group)
    inp = W.make_layer(wl, 0, "cuda")
    run_and_check(wl, inp, host(inp), tag=f"group {group}")
