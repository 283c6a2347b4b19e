"""Parity of the cache update after acceptance (Algorithm 2, Update; bd_advance) with the
oracle, and a multi-step loop in which carry-mode selection runs on the slid window and
must keep matching the oracle's selection recomputed from scratch at each new length."""

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from tests.parity import check_attention, check_selection, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def bf16_randn(g, *shape):
    return torch.randn(*shape, generator=g).to(torch.bfloat16)


@pytest.mark.parametrize("n_acc,window,n_q", [([4, 2, 5], 32, 6), ([5, 5, 5], 32, 6), ([0, 3, 1], 32, 6),
                                               ([5, 5, 5], 4, 6), ([9, 7, 8], 16, 6)])
def test_advance_matches_oracle(n_acc, window, n_q):
    b, hq, hkv, d, t, cap = 3, 8, 2, 128, 500, 40
    g = torch.Generator().manual_seed(3 + window + sum(n_acc))
    q_win, q_ver = bf16_randn(g, b, hq, window, d), bf16_randn(g, b, hq, n_q, d)
    lse_win, lse_ver = torch.randn(b, hq, window, generator=g), torch.randn(b, hq, n_q, generator=g)
    count = torch.tensor([[30, 38], [0, 39], [12, 34]], dtype=torch.int32)   # some units without room
    idx = torch.full((b, hkv, cap), -1, dtype=torch.int32)
    for bi in range(b):
        for kv in range(hkv):
            c = int(count[bi, kv])
            idx[bi, kv, :c] = torch.sort(torch.randperm(t, generator=g)[:c]).values.int()
    dev = {k: v.cuda() for k, v in dict(q_win=q_win, q_ver=q_ver, lse_win=lse_win, lse_ver=lse_ver, idx=idx,
                                        count=count).items()}
    n_dev = torch.tensor(n_acc, dtype=torch.int32, device="cuda")
    out = torch.zeros(b, dtype=torch.int32, device="cuda")
    shape = bd.make_shape(b, hq, hkv, d, t, t + n_q)
    bd.bd_advance(shape, window, n_q, n_dev, dev["q_ver"], dev["lse_ver"], dev["q_win"], dev["lse_win"], dev["idx"],
                  dev["count"], out)
    torch.cuda.synchronize()
    a = oracle.batch_advance(np.array(n_acc), n_q)
    assert out.cpu().tolist() == [a] * b
    q_ref, l_ref = oracle.advance_window(f64(q_win), lse_win.double().numpy(), f64(q_ver), lse_ver.double().numpy(), a)
    assert np.array_equal(f64(dev["q_win"]), q_ref)                     # a copy: bit-exact
    assert np.array_equal(dev["lse_win"].cpu().double().numpy(), l_ref)
    i_ref, c_ref, full = oracle.append_view(idx.numpy(), count.numpy(), t, a, cap)
    assert full == bool(((count + a) > cap).any())
    assert dev["idx"].cpu().numpy().tolist() == i_ref.tolist()
    assert dev["count"].cpu().numpy().tolist() == c_ref.tolist()


def test_multistep_carry_selection_on_the_slid_window():
    """Three steps of select (carry mode) -> verify -> accept counts -> advance, each with the
    context grown by the settled rows; the window and its LSE are only ever slid, never
    recomputed, and selection still matches the oracle's from-scratch selection."""
    b, hq, hkv, d, W, gamma = 2, 8, 2, 128, 32, 5
    t0, steps, budget, sink, recent = 3000, 3, 256, 4, 64
    cap = t0 + steps * (gamma + 1)
    g = torch.Generator().manual_seed(77)
    K, V = bf16_randn(g, b, hkv, cap, d).cuda(), bf16_randn(g, b, hkv, cap, d).cuda()
    q_all = bf16_randn(g, b, hq, cap, d).cuda()                        # the query of every position
    Kh = f64(K)
    qh = f64(q_all)
    rng = np.random.default_rng(5)
    t = t0
    q_win = q_all[:, :, t - W: t].clone()
    sh = bd.make_shape(b, hq, hkv, d, t - W, cap)
    lse_win = torch.empty(b, hq, W, dtype=torch.float32, device="cuda")
    ws0 = bd.Workspace(bd.bd_workspace_size(sh, bd.BD_OP_VERIFY, 1, W))
    bd.bd_verify_attn(sh, q_win, W, K, None, None, lse_win, ws0)
    idx = torch.empty(b, hkv, budget, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, hkv, dtype=torch.int32, device="cuda")
    vo = torch.empty(b, hq, gamma + 1, d, dtype=torch.bfloat16, device="cuda")
    vl = torch.empty(b, hq, gamma + 1, dtype=torch.float32, device="cuda")
    adv = torch.zeros(b, dtype=torch.int32, device="cuda")
    for step in range(steps):
        shape = bd.make_shape(b, hq, hkv, d, t, cap)
        ws = bd.Workspace.for_step(shape, budget, W, gamma)
        bd.bd_select_budget(shape, K, q_win, lse_win, W, budget, sink, recent, 1, idx, cnt, ws)
        lse_ref = oracle.window_lse(qh[:, :, t - W: t], Kh, t)
        score_ref = oracle.window_scores(qh[:, :, t - W: t], Kh, lse_ref, t)
        idx_ref = np.full((b, hkv, budget), -1)
        cnt_ref = np.zeros((b, hkv), dtype=np.int64)
        for bi in range(b):
            for kv in range(hkv):
                keep = oracle.select_from_scores(score_ref[bi, kv], t, budget, sink, recent, 1)
                idx_ref[bi, kv, :keep.size] = keep
                cnt_ref[bi, kv] = keep.size
        torch.cuda.synchronize()
        check_selection(idx, cnt, idx_ref, cnt_ref, score_ref, t, budget, sink, recent, 1, what=f"step {step}")
        q_ver = q_all[:, :, t: t + gamma + 1].contiguous()
        bd.bd_verify_attn(shape, q_ver, gamma + 1, K, V, vo, vl, ws)
        o_ref, l_ref = oracle.verify_attn(qh[:, :, t: t + gamma + 1], Kh, f64(V), t)
        torch.cuda.synchronize()
        check_attention(vo, vl, o_ref, l_ref, f"step {step} verify")
        n_acc = rng.integers(1, gamma + 1, size=b)
        bd.bd_advance(shape, W, gamma + 1, torch.from_numpy(n_acc).int().cuda(), q_ver, vl, q_win, lse_win, None,
                      None, adv)
        torch.cuda.synchronize()
        a = int(adv[0].item())
        assert a == oracle.batch_advance(n_acc, gamma + 1)
        t += a
        assert torch.equal(q_win, q_all[:, :, t - W: t])
        err = np.abs(lse_win.cpu().double().numpy() - oracle.window_lse(qh[:, :, t - W: t], Kh, t)).max()
        assert err <= 1e-3, f"step {step}: slid window LSE off by {err}"
        assert ws.status() == 0


def test_amortised_loop_view_grows_by_the_settled_rows():
    """Algorithm 2 as written: sparsify once, then every step appends its settled rows to the
    drafter's view.  After each advance the next step's draft pass must equal the oracle's
    draft attention over (first selection + every appended position)."""
    b, hq, hkv, d, W, gamma = 2, 8, 2, 128, 32, 3
    t0, steps, budget, sink, recent = 2000, 3, 128, 4, 32
    cap_rows = t0 + steps * (gamma + 1)
    capacity = budget + steps * (gamma + 1)
    g = torch.Generator().manual_seed(91)
    K, V = bf16_randn(g, b, hkv, cap_rows, d).cuda(), bf16_randn(g, b, hkv, cap_rows, d).cuda()
    q_all = bf16_randn(g, b, hq, cap_rows, d).cuda()
    qd_all = bf16_randn(g, steps, gamma, b, hq, d).cuda()          # drafter queries of every pass
    Kh, Vh = f64(K), f64(V)
    rng = np.random.default_rng(8)
    t = t0
    shape = bd.make_shape(b, hq, hkv, d, t, cap_rows)
    idx = torch.full((b, hkv, capacity), -1, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, hkv, dtype=torch.int32, device="cuda")
    ws = bd.Workspace.for_step(shape, budget, W, gamma)
    q_win = q_all[:, :, t - W: t].contiguous()
    sel = torch.full((b, hkv, budget), -1, dtype=torch.int32, device="cuda")
    bd.bd_select_budget(shape, K, q_win, None, W, budget, sink, recent, 1, sel, cnt, ws)
    idx[:, :, :budget] = sel
    lse_win = torch.empty(b, hq, W, dtype=torch.float32, device="cuda")
    vo = torch.empty(b, hq, gamma + 1, d, dtype=torch.bfloat16, device="cuda")
    vl = torch.empty(b, hq, gamma + 1, dtype=torch.float32, device="cuda")
    do = torch.empty(b, hq, d, dtype=torch.bfloat16, device="cuda")
    dl = torch.empty(b, hq, dtype=torch.float32, device="cuda")
    adv = torch.zeros(b, dtype=torch.int32, device="cuda")
    for step in range(steps):
        shape = bd.make_shape(b, hq, hkv, d, t, cap_rows)
        ws = bd.Workspace.for_step(shape, capacity, W, gamma)
        torch.cuda.synchronize()
        idx_h, cnt_h = idx.cpu().numpy(), cnt.cpu().numpy()
        for j in range(gamma):
            q = qd_all[step, j].contiguous()
            bd.bd_draft_attn(shape, q, K, V, idx, cnt, capacity, j, do, dl, ws)
            o_ref, l_ref = oracle.draft_attn(f64(q), Kh, Vh, idx_h, cnt_h, t, j)
            torch.cuda.synchronize()
            check_attention(do, dl, o_ref, l_ref, f"step {step} draft {j}")
        q_ver = q_all[:, :, t: t + gamma + 1].contiguous()
        bd.bd_verify_attn(shape, q_ver, gamma + 1, K, V, vo, vl, ws)
        n_acc = rng.integers(0, gamma + 1, size=b)
        bd.bd_advance(shape, W, gamma + 1, torch.from_numpy(n_acc).int().cuda(), q_ver, vl, q_win, lse_win, idx,
                      cnt, adv)
        torch.cuda.synchronize()
        a = int(adv[0].item())
        i_ref, c_ref, full = oracle.append_view(idx_h, cnt_h, t, a, capacity)
        assert not full
        assert idx.cpu().numpy().tolist() == i_ref.tolist() and cnt.cpu().numpy().tolist() == c_ref.tolist()
        t += a
        assert ws.status() == 0
