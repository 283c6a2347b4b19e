"""The library's planners accept every synthetic workload (CPU, no device: the plans are
made for one SM, the most demanding split): bd_workspace_size is nonzero for the selection
(its size covers the window LSE computed in the call as well), the drafter passes and the
verify block of each workload and each budget of the 16K sweep."""

import ctypes

import pytest

import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import workload as W


@pytest.fixture(scope="module")
def lib():
    bd.build()
    return bd.library()


def cases():
    for name, wl in W.WORKLOADS.items():
        yield name, wl
    for budget in W.SWEEP_16K:
        yield f"l8b_16k_b8@B{budget}", W.WORKLOADS["l8b_16k_b8"].with_budget(budget)


@pytest.mark.parametrize("name,wl", list(cases()), ids=[c[0] for c in cases()])
def test_every_workload_is_planned(lib, name, wl):
    s = bd.make_shape(wl.batch, wl.h_q, wl.h_kv, wl.head_dim, wl.t_ctx, wl.t_cap)
    size = lambda op, budget, n_q: lib.bd_workspace_size(ctypes.byref(s), op, budget, n_q)
    assert size(bd.BD_OP_SELECT, wl.budget, wl.window) > 0
    assert size(bd.BD_OP_DRAFT, wl.budget, wl.gamma) > 0
    assert size(bd.BD_OP_VERIFY, wl.budget, wl.gamma + 1) > 0
