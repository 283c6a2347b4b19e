"""HostStepIO (pinned host buffers, packed transfers on a side stream, double buffering)
gives exactly the results of SpecStep run directly on device tensors, step by step,
eagerly and inside a CUDA graph."""

import pytest
import torch

import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def _inputs(wl, base, other):
    """Per-step inputs: the queries and block rows of `other`, over the context of `base`."""
    g1 = wl.gamma + 1
    return dict(q_win=other.q_win, q_draft=other.q_draft, q_verify=other.q_verify,
                k_rows=other.k_cache[:, :, wl.t_ctx: wl.t_ctx + g1].clone(),
                v_rows=other.v_cache[:, :, wl.t_ctx: wl.t_ctx + g1].clone())


def _reference(wl, base, inp, lse):
    g1 = wl.gamma + 1
    k, v = base.k_cache.clone(), base.v_cache.clone()
    k[:, :, wl.t_ctx: wl.t_ctx + g1] = inp["k_rows"]
    v[:, :, wl.t_ctx: wl.t_ctx + g1] = inp["v_rows"]
    st = bd.SpecStep.for_workload(wl)
    st.run(k, v, inp["q_win"], inp["q_draft"], inp["q_verify"], lse)
    torch.cuda.synchronize()
    return dict(idx=st.idx.cpu(), count=st.count.cpu(), draft_o=st.draft_o.cpu(), draft_lse=st.draft_lse.cpu(),
                verify_o=st.verify_o.cpu(), verify_lse=st.verify_lse.cpu())


@pytest.mark.parametrize("graph", [False, True])
def test_host_step_io_matches_spec_step(graph):
    wl = W.WORKLOADS["l8b_4k"]
    base = W.make_layer(wl, 0, "cuda")
    other = W.make_layer(wl, 0, "cuda", first_seq=100)
    ins = [_inputs(wl, base, base), _inputs(wl, base, other)]
    probe = bd.SpecStep.for_workload(wl)
    lses = [probe.window_lse(base.k_cache, x["q_win"]) for x in ins]
    refs = [_reference(wl, base, x, l) for x, l in zip(ins, lses)]

    k, v = base.k_cache.clone(), base.v_cache.clone()
    st = bd.SpecStep.for_workload(wl)
    io = bd.HostStepIO([(st, k, v, True)])
    for slot in range(2):
        h = io.host_inputs(slot)
        for name in ("q_win", "q_draft", "q_verify", "k_rows", "v_rows"):
            h[name + "0"].copy_(ins[slot][name])
        h["lse0"].copy_(lses[slot])
    torch.cuda.synchronize()
    if graph:
        io.run(2)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                io.run(5)
        torch.cuda.current_stream().wait_stream(s)
        g.replay()
    else:
        io.run(5)
    torch.cuda.synchronize()
    for slot in range(2):
        out = io.host_outputs(slot)
        for name, want in refs[slot].items():
            assert torch.equal(out[name + "0"], want), f"slot {slot}: {name}"
    assert io.bytes_in > 0 and io.bytes_out > 0
    assert st.ws.status() == 0
