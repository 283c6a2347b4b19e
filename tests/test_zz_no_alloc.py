"""The allocation-free draft entry point (bd_draft_attn_static) against bd_draft_attn.

Some callers cannot allocate device memory when they call the library (a plugin handed
only a stream and tensor pointers, a serving loop whose memory is fixed after start-up).
bd_draft_attn_static serves them with scratch from the library's own device array.  This
test calls it through the C ABI twice in a row, with different queries and passes so that
stale scratch from the first call would show, and checks each result against the
workspace entry point's on the same inputs, within the parity tolerance.
"""

import pytest
import torch

import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W
from tests.parity import check_attention, f64

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("budget", [512, 2048])
def test_draft_attn_static_matches_workspace_entry_point(budget):
    """budget 2048: every CTA of a unit's cluster gathers several tiles."""
    bd.build()
    wl = W.WORKLOADS["l8b_16k_b8"]
    inp = W.make_layer(wl, 0, "cuda")
    st = bd.SpecStep.for_workload(wl, budget=budget, n_recent=budget // 4)
    st.select(inp.k_cache, inp.q_win, None)                 # a real sparse view to gather
    o = torch.empty(wl.batch, wl.h_q, wl.head_dim, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(wl.batch, wl.h_q, device="cuda")
    for j in (wl.gamma - 1, 0):                              # two calls in a row
        st.draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache)
        bd.bd_draft_attn_static(st.shape, inp.q_draft[j], inp.k_cache, inp.v_cache, st.idx, st.count,
                                st.budget, j, o, lse)
        torch.cuda.synchronize()
        check_attention(o, lse, f64(st.draft_o[j]), f64(st.draft_lse[j]), f"static draft B={budget} j={j}")
    assert st.ws.status() == 0


def test_draft_attn_static_rejects_oversized_scratch():
    bd.build()
    # 4 MiB is enough for the counters of ~1M (sequence, KV head) units but not 2M
    shape = bd.make_shape(batch=4096, h_q=4096, h_kv=512, head_dim=128, t_ctx=64, t_cap=80)
    dummy = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(bd.BudgetDraftError) as e:
        bd.bd_draft_attn_static(shape, dummy, dummy, dummy, dummy, dummy, 8, 0, dummy, None)
    assert e.value.status == -4                              # BD_ERR_WORKSPACE
