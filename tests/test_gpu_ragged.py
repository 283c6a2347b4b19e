"""Per-sequence context lengths (bd_shape.seq_lens): every call against the oracle run
sequence by sequence at that sequence's own length, the keep-all rule for a sequence that
fits the budget, ragged block-row writes, and a multi-step loop in which every sequence
advances by its own accepted count on the device."""

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as wk
from tests.parity import check_attention, check_selection, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def bf16_randn(g, *shape):
    return torch.randn(*shape, generator=g).to(torch.bfloat16)


def oracle_selection(qw, K, lse, t, budget, sink, recent):
    score = oracle.window_scores(qw, K, lse, t)
    h_kv = K.shape[1]
    idx = np.full((1, h_kv, budget), -1)
    cnt = np.zeros((1, h_kv), dtype=np.int64)
    for kv in range(h_kv):
        keep = oracle.select_from_scores(score[0, kv], t, budget, sink, recent, 1)
        idx[0, kv, :keep.size] = keep
        cnt[0, kv] = keep.size
    return idx, cnt, score


@pytest.mark.parametrize("mode", ["carry", "self"])
def test_ragged_lengths_match_per_sequence_oracle(mode):
    lens = [3000, 2433, 1777, 200]                 # the last one fits the budget: keep all
    b, hq, hkv, d, W, gamma, budget, sink, recent = len(lens), 8, 2, 128, 32, 3, 256, 4, 64
    t_max = max(lens)
    wl = wk.tiny_workload(batch=b, h_q=hq, h_kv=hkv, head_dim=d, t_ctx=t_max, budget=budget, n_sink=sink,
                         n_recent=recent, window=W, gamma=gamma)
    inp = wk.make_layer(wl, 0, "cuda")
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    shape = bd.make_shape(b, hq, hkv, d, t_max, wl.t_cap, seq_lens=lens_d)
    h = dict(K=f64(inp.k_cache), V=f64(inp.v_cache), QW=f64(inp.q_win), QD=f64(inp.q_draft), QV=f64(inp.q_verify))
    lse_ref = [oracle.window_lse(h["QW"][i:i + 1], h["K"][i:i + 1], lens[i]) for i in range(b)]
    lse_d = torch.from_numpy(np.concatenate(lse_ref)).float().cuda() if mode == "carry" else None
    ws = bd.Workspace.for_step(shape, budget, W, gamma)
    idx = torch.empty(b, hkv, budget, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, hkv, dtype=torch.int32, device="cuda")
    idx_ref = np.full((b, hkv, budget), -1)
    cnt_ref = np.zeros((b, hkv), dtype=np.int64)
    refs = []
    for i, t in enumerate(lens):
        ir, cr, score = oracle_selection(h["QW"][i:i + 1], h["K"][i:i + 1], lse_ref[i], t, budget, sink, recent)
        idx_ref[i], cnt_ref[i] = ir[0], cr[0]
        refs.append((ir, cr, score))
    # carry mode also with BD_SELECT_WINDOW_READY: the tile layout of the lengths is then
    # built before the dependency wait
    for flags in ((0, bd.BD_SELECT_WINDOW_READY) if mode == "carry" else (0,)):
        idx.fill_(-7)
        bd.bd_select_budget(shape, inp.k_cache, inp.q_win, lse_d, W, budget, sink, recent, 1, idx, cnt, ws,
                            flags=flags)
        torch.cuda.synchronize()
        for i, t in enumerate(lens):
            ir, cr, score = refs[i]
            check_selection(idx[i:i + 1], cnt[i:i + 1], ir, cr, score, t, budget, sink, recent, 1,
                            what=f"{mode} flags {flags} seq {i} T={t}")
    assert cnt_ref[-1].tolist() == [lens[-1]] * hkv             # B >= T_b keeps everything
    # drafts on the oracle's selection, verify
    idx.copy_(torch.from_numpy(idx_ref).int())
    cnt.copy_(torch.from_numpy(cnt_ref).int())
    o = torch.empty(b, hq, d, dtype=torch.bfloat16, device="cuda")
    l = torch.empty(b, hq, dtype=torch.float32, device="cuda")
    for j in range(gamma):
        bd.bd_draft_attn(shape, inp.q_draft[j], inp.k_cache, inp.v_cache, idx, cnt, budget, j, o, l, ws)
        torch.cuda.synchronize()
        for i, t in enumerate(lens):
            o_ref, l_ref = oracle.draft_attn(h["QD"][j][i:i + 1], h["K"][i:i + 1], h["V"][i:i + 1],
                                             idx_ref[i:i + 1], cnt_ref[i:i + 1], t, j)
            check_attention(o[i:i + 1], l[i:i + 1], o_ref, l_ref, f"draft j={j} seq {i} T={t}")
    vo = torch.empty(b, hq, gamma + 1, d, dtype=torch.bfloat16, device="cuda")
    vl = torch.empty(b, hq, gamma + 1, dtype=torch.float32, device="cuda")
    bd.bd_verify_attn(shape, inp.q_verify, gamma + 1, inp.k_cache, inp.v_cache, vo, vl, ws)
    torch.cuda.synchronize()
    for i, t in enumerate(lens):
        o_ref, l_ref = oracle.verify_attn(h["QV"][i:i + 1], h["K"][i:i + 1], h["V"][i:i + 1], t)
        check_attention(vo[i:i + 1], vl[i:i + 1], o_ref, l_ref, f"verify seq {i} T={t}")
    assert ws.status() == 0


def test_ragged_window_lse_matches_oracle():
    """SpecStep.window_lse with per-sequence lengths: each sequence's window rows over its own
    causal prefix (the carried state a prefill leaves for carry mode)."""
    lens = [3000, 2433, 1777, 200]
    b, hq, hkv, d, W = len(lens), 8, 2, 128, 32
    wl = wk.tiny_workload(batch=b, h_q=hq, h_kv=hkv, head_dim=d, t_ctx=max(lens), budget=256, n_sink=4,
                         n_recent=64, window=W, gamma=3)
    inp = wk.make_layer(wl, 0, "cuda")
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    st = bd.SpecStep(b, hq, hkv, d, wl.t_ctx, wl.t_cap, 256, 4, 64, W, 3, seq_lens=lens_d)
    lse = st.window_lse(inp.k_cache, inp.q_win)
    torch.cuda.synchronize()
    K, QW = f64(inp.k_cache), f64(inp.q_win)
    for i, t in enumerate(lens):
        ref = oracle.window_lse(QW[i:i + 1], K[i:i + 1], t)
        err = np.abs(f64(lse[i:i + 1]) - ref).max()
        assert err <= 1e-3, f"seq {i} T={t}: window lse err {err:.3e}"


def test_ragged_block_rows_land_at_each_sequence_length():
    lens = [50, 37, 64]
    b, hkv, d, n_rows, t_cap = len(lens), 2, 64, 4, 80
    g = torch.Generator().manual_seed(4)
    K, V = bf16_randn(g, b, hkv, t_cap, d).cuda(), bf16_randn(g, b, hkv, t_cap, d).cuda()
    K0, V0 = K.clone(), V.clone()
    kr = bf16_randn(g, b, hkv, n_rows, d).pin_memory()          # straight from pinned host memory
    vr = bf16_randn(g, b, hkv, n_rows, d).pin_memory()
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    shape = bd.make_shape(b, 4, hkv, d, max(lens), t_cap, seq_lens=lens_d)
    bd.bd_write_block_rows(shape, n_rows, kr, vr, K, V)
    torch.cuda.synchronize()
    for i, t in enumerate(lens):
        K0[i, :, t: t + n_rows] = kr[i].cuda()
        V0[i, :, t: t + n_rows] = vr[i].cuda()
    assert torch.equal(K, K0) and torch.equal(V, V0)


def test_ragged_multistep_each_sequence_advances_by_its_own_count():
    """Three steps: carry-mode selection on the slid windows, verify, per-sequence accepted
    counts, bd_advance updating the lengths on the device; each sequence's selection and
    window LSE must match the oracle at that sequence's own new length."""
    lens0 = [2500, 2100, 2777]
    b, hq, hkv, d, W, gamma, budget, sink, recent = len(lens0), 8, 2, 128, 32, 5, 200, 4, 48
    steps = 3
    cap = max(lens0) + steps * (gamma + 1) + 1
    g = torch.Generator().manual_seed(12)
    K, V = bf16_randn(g, b, hkv, cap, d).cuda(), bf16_randn(g, b, hkv, cap, d).cuda()
    q_all = bf16_randn(g, b, hq, cap, d).cuda()
    Kh, qh = f64(K), f64(q_all)
    lens = list(lens0)
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    t_max_cap = cap - (gamma + 1)
    q_win = torch.stack([q_all[i, :, lens[i] - W: lens[i]] for i in range(b)]).contiguous()
    lse_win = torch.from_numpy(np.concatenate([oracle.window_lse(qh[i:i + 1, :, lens[i] - W: lens[i]], Kh[i:i + 1],
                                                                 lens[i]) for i in range(b)])).float().cuda()
    idx = torch.empty(b, hkv, budget, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, hkv, dtype=torch.int32, device="cuda")
    vo = torch.empty(b, hq, gamma + 1, d, dtype=torch.bfloat16, device="cuda")
    vl = torch.empty(b, hq, gamma + 1, dtype=torch.float32, device="cuda")
    adv = torch.zeros(b, dtype=torch.int32, device="cuda")
    rng = np.random.default_rng(3)
    for step in range(steps):
        shape = bd.make_shape(b, hq, hkv, d, t_max_cap, cap, seq_lens=lens_d)
        ws = bd.Workspace.for_step(shape, budget, W, gamma)
        bd.bd_select_budget(shape, K, q_win, lse_win, W, budget, sink, recent, 1, idx, cnt, ws)
        torch.cuda.synchronize()
        for i, t in enumerate(lens):
            lr = oracle.window_lse(qh[i:i + 1, :, t - W: t], Kh[i:i + 1], t)
            ir, cr, score = oracle_selection(qh[i:i + 1, :, t - W: t], Kh[i:i + 1], lr, t, budget, sink, recent)
            check_selection(idx[i:i + 1], cnt[i:i + 1], ir, cr, score, t, budget, sink, recent, 1,
                            what=f"step {step} seq {i} T={t}")
        q_ver = torch.stack([q_all[i, :, lens[i]: lens[i] + gamma + 1] for i in range(b)]).contiguous()
        bd.bd_verify_attn(shape, q_ver, gamma + 1, K, V, vo, vl, ws)
        n_acc = rng.integers(0, gamma + 1, size=b)
        bd.bd_advance(shape, W, gamma + 1, torch.from_numpy(n_acc).int().cuda(), q_ver, vl, q_win, lse_win, None,
                      None, adv)
        torch.cuda.synchronize()
        a = [int(x) + 1 for x in n_acc]
        assert adv.cpu().tolist() == a
        lens = [t + ai for t, ai in zip(lens, a)]
        assert lens_d.cpu().tolist() == lens                        # advanced on the device
        for i, t in enumerate(lens):
            assert torch.equal(q_win[i], q_all[i, :, t - W: t])
            err = np.abs(lse_win[i].cpu().double().numpy()
                         - oracle.window_lse(qh[i:i + 1, :, t - W: t], Kh[i:i + 1], t)[0]).max()
            assert err <= 1e-3, f"step {step} seq {i}: slid window LSE off by {err}"
        assert ws.status() == 0


@pytest.mark.parametrize("mode", ["carry", "self"])
def test_ragged_mha_batch_beyond_1024_units(mode):
    """The paper's verifier is multi-head (one query head per KV head: 32 KV heads at d 128),
    so a ragged batch of 40 sequences already holds 1280 (sequence, KV head) units, more than
    a table of 1024 would: selection, a draft pass and the verify, each against the oracle
    on a sample of sequences at their own lengths."""
    b, hq, hkv, d, W, gamma, budget, sink, recent = 40, 32, 32, 128, 32, 3, 128, 4, 16
    g = torch.Generator().manual_seed(40)
    lens = torch.randint(300, 901, (b,), generator=g).tolist()
    lens[-1] = 100                                   # fits the budget: keep all
    t_max = max(lens)
    wl = wk.tiny_workload(batch=b, h_q=hq, h_kv=hkv, head_dim=d, t_ctx=t_max, budget=budget, n_sink=sink,
                         n_recent=recent, window=W, gamma=gamma)
    inp = wk.make_layer(wl, 0, "cuda")
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    shape = bd.make_shape(b, hq, hkv, d, t_max, wl.t_cap, seq_lens=lens_d)
    sample = [0, 7, 19, 33, b - 1]
    h = {i: dict(K=f64(inp.k_cache[i:i + 1]), V=f64(inp.v_cache[i:i + 1]), QW=f64(inp.q_win[i:i + 1]),
                 QD=f64(inp.q_draft[:, i:i + 1]), QV=f64(inp.q_verify[i:i + 1])) for i in sample}
    lse_ref = {i: oracle.window_lse(h[i]["QW"], h[i]["K"], lens[i]) for i in sample}
    if mode == "carry":   # the carried LSE of the unsampled sequences comes from the library's own pass
        st = bd.SpecStep(b, hq, hkv, d, t_max, wl.t_cap, budget, sink, recent, W, gamma, seq_lens=lens_d)
        lse_d = st.window_lse(inp.k_cache, inp.q_win)
        for i in sample:
            lse_d[i:i + 1] = torch.from_numpy(lse_ref[i]).float().cuda()
    else:
        lse_d = None
    ws = bd.Workspace.for_step(shape, budget, W, gamma)
    idx = torch.empty(b, hkv, budget, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, hkv, dtype=torch.int32, device="cuda")
    bd.bd_select_budget(shape, inp.k_cache, inp.q_win, lse_d, W, budget, sink, recent, 1, idx, cnt, ws)
    torch.cuda.synchronize()
    refs = {}
    for i in sample:
        ir, cr, score = oracle_selection(h[i]["QW"], h[i]["K"], lse_ref[i], lens[i], budget, sink, recent)
        refs[i] = (ir, cr)
        check_selection(idx[i:i + 1], cnt[i:i + 1], ir, cr, score, lens[i], budget, sink, recent, 1,
                        what=f"{mode} seq {i} T={lens[i]}")
    assert int(cnt[b - 1, 0]) == lens[-1]
    for i in sample:   # the drafts run on the oracle's view of the sampled sequences
        idx[i] = torch.from_numpy(refs[i][0][0]).int().cuda()
        cnt[i] = torch.from_numpy(refs[i][1][0]).int().cuda()
    o = torch.empty(b, hq, d, dtype=torch.bfloat16, device="cuda")
    l = torch.empty(b, hq, dtype=torch.float32, device="cuda")
    bd.bd_draft_attn(shape, inp.q_draft[1], inp.k_cache, inp.v_cache, idx, cnt, budget, 1, o, l, ws)
    vo = torch.empty(b, hq, gamma + 1, d, dtype=torch.bfloat16, device="cuda")
    vl = torch.empty(b, hq, gamma + 1, dtype=torch.float32, device="cuda")
    bd.bd_verify_attn(shape, inp.q_verify, gamma + 1, inp.k_cache, inp.v_cache, vo, vl, ws)
    torch.cuda.synchronize()
    for i in sample:
        o_ref, l_ref = oracle.draft_attn(h[i]["QD"][1], h[i]["K"], h[i]["V"], refs[i][0], refs[i][1], lens[i], 1)
        check_attention(o[i:i + 1], l[i:i + 1], o_ref, l_ref, f"{mode} draft seq {i} T={lens[i]}")
        o_ref, l_ref = oracle.verify_attn(h[i]["QV"], h[i]["K"], h[i]["V"], lens[i])
        check_attention(vo[i:i + 1], vl[i:i + 1], o_ref, l_ref, f"{mode} verify seq {i} T={lens[i]}")
    assert ws.status() == 0
