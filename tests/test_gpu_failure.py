"""The device-side error path without a GPU fault: a bounded wait that runs out (on a
barrier nothing completes) records BD_ERR_TIMEOUT in the workspace status word, the host
reads it, and the context stays usable for the next call."""

import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W
from tests.parity import check_attention, f64

pytestmark = pytest.mark.gpu
TIMEOUT = -6


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def test_bounded_wait_reports_timeout_and_context_survives():
    ws = bd.Workspace(1024)
    bd.bd_check_wait_timeout(ws, 2000)            # 2 ms on a barrier nothing completes
    assert ws.status() == TIMEOUT
    assert ws.status() == 0                       # reading clears the word
    # the next real call on the same context works and reports no error
    wl = W.WORKLOADS["tiny_1k"]
    inp = W.make_layer(wl, 0, "cuda")
    st = bd.SpecStep.for_workload(wl)
    st.verify(inp.q_verify, inp.k_cache, inp.v_cache)
    o_ref, l_ref = oracle.verify_attn(f64(inp.q_verify), f64(inp.k_cache), f64(inp.v_cache), wl.t_ctx)
    torch.cuda.synchronize()
    check_attention(st.verify_o, st.verify_lse, o_ref, l_ref, "verify after the timeout probe")
    assert st.ws.status() == 0
