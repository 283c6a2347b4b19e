"""The allocation-free draft entry point (bd_draft_attn_static) against the fp64 oracle.

Some callers cannot allocate device memory when they call the library (a plugin handed
only a stream and tensor pointers, a serving loop whose memory is fixed after start-up).
bd_draft_attn_static serves them with scratch from the library's own device array.  This
test calls it through the C ABI twice in a row, with different queries and passes so that
stale scratch from the first call would show, and checks each result against
oracle.draft_attn on the same inputs, within the parity tolerance, and against the
workspace entry point bd_draft_attn.  The sparse view is a seeded random subset drawn on
the host, so the oracle's inputs come from the input generators alone.
"""

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W
from tests.parity import check_attention, f64

pytestmark = pytest.mark.gpu


def seeded_view(wl, budget, seed):
    """Ascending distinct positions of [0, t_ctx) per (sequence, KV head), budget of them."""
    rng = np.random.default_rng(seed)
    idx = np.stack([np.sort(rng.choice(wl.t_ctx, budget, replace=False))
                    for _ in range(wl.batch * wl.h_kv)]).reshape(wl.batch, wl.h_kv, budget)
    count = np.full((wl.batch, wl.h_kv), budget, dtype=np.int64)
    return idx, count


@pytest.mark.parametrize("budget", [512, 2048])
def test_draft_attn_static_matches_oracle(budget):
    """budget 2048: every CTA of a unit's cluster gathers several tiles."""
    bd.build()
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    idx_h, cnt_h = seeded_view(wl, budget, 7000 + budget)
    K, V, QD = f64(inp.k_cache), f64(inp.v_cache), f64(inp.q_draft)
    st = bd.SpecStep.for_workload(wl, budget=budget, n_recent=budget // 4)
    st.idx.copy_(torch.from_numpy(idx_h).int())
    st.count.copy_(torch.from_numpy(cnt_h).int())
    o = torch.empty(wl.batch, wl.h_q, wl.head_dim, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(wl.batch, wl.h_q, device="cuda")
    for j in (wl.gamma - 1, 0):                              # two calls in a row
        bd.bd_draft_attn_static(st.shape, inp.q_draft[j], inp.k_cache, inp.v_cache, st.idx, st.count,
                                st.budget, j, o, lse)
        st.draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache)
        torch.cuda.synchronize()
        o_ref, l_ref = oracle.draft_attn(QD[j], K, V, idx_h, cnt_h, wl.t_ctx, j)
        check_attention(o, lse, o_ref, l_ref, f"static draft B={budget} j={j}")
        check_attention(o, lse, f64(st.draft_o[j]), f64(st.draft_lse[j]), f"static vs workspace B={budget} j={j}")
    assert st.ws.status() == 0


def test_draft_attn_static_reports_device_errors_until_read():
    """The array's status word keeps a device-side error of a static call (an index past the
    context, skipped like in bd_draft_attn) until bd_draft_static_status reads and clears it;
    clean calls leave it at zero."""
    bd.build()
    wl = W.tiny_workload(batch=1, h_q=4, h_kv=1, head_dim=64, t_ctx=100, budget=8)
    inp = W.make_layer(wl, 0, "cuda")
    st = bd.SpecStep.for_workload(wl)
    o = torch.empty(1, 4, 64, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(1, 4, device="cuda")
    st.count.fill_(4)
    assert bd.bd_draft_static_status() in (0, -1)          # whatever earlier calls left, now cleared
    st.idx.copy_(torch.tensor([[[0, 5, 9, 20, -1, -1, -1, -1]]], dtype=torch.int32))
    bd.bd_draft_attn_static(st.shape, inp.q_draft[0], inp.k_cache, inp.v_cache, st.idx, st.count, 8, 0, o, lse)
    assert bd.bd_draft_static_status() == 0
    st.idx.copy_(torch.tensor([[[0, 5, 100000, 20, -1, -1, -1, -1]]], dtype=torch.int32))
    bd.bd_draft_attn_static(st.shape, inp.q_draft[0], inp.k_cache, inp.v_cache, st.idx, st.count, 8, 0, o, lse)
    st.idx.copy_(torch.tensor([[[0, 5, 9, 20, -1, -1, -1, -1]]], dtype=torch.int32))
    bd.bd_draft_attn_static(st.shape, inp.q_draft[0], inp.k_cache, inp.v_cache, st.idx, st.count, 8, 0, o, lse)
    assert bd.bd_draft_static_status() == -1                # BD_ERR_INVALID_ARG, kept across the clean call
    assert bd.bd_draft_static_status() == 0                 # reading clears it


def test_draft_attn_static_rejects_oversized_scratch():
    bd.build()
    # 4 MiB is enough for the counters of ~1M (sequence, KV head) units but not 2M
    shape = bd.make_shape(batch=4096, h_q=4096, h_kv=512, head_dim=128, t_ctx=64, t_cap=80)
    dummy = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(bd.BudgetDraftError) as e:
        bd.bd_draft_attn_static(shape, dummy, dummy, dummy, dummy, dummy, 8, 0, dummy, None)
    assert e.value.status == -4                              # BD_ERR_WORKSPACE
