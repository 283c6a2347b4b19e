"""bench.py's algorithmic byte accounting (the numerator of every GB/s and roofline figure)
against the per-workload totals the measurement plan fixes independently: what the method
must read per step (middle keys once for the selection, the sparse view once plus the
drafted rows, the whole cache for the verify), in MiB for the single-layer workloads and
GB for the 32-layer stack.  CPU only."""

import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2606_00144_gb300 import workload as W  # noqa: E402

MIB = 1 << 20


@pytest.mark.parametrize("name,budget,n_recent,mib", [
    ("tiny_1k", 256, 64, 0.9),
    ("l8b_4k", 512, 128, 25.8),
    ("l8b_8k_b4", 1024, 256, 206.0),
    ("l8b_16k_b8", 256, 64, 775.0),
    ("l8b_16k_b8", 512, 128, 782.0),
    ("l8b_16k_b8", 1024, 256, 796.0),
    ("l8b_16k_b8", 2048, 512, 824.0),
    ("l8b_16k_b8", 16384, 4096, 1024.0),
])
def test_single_layer_totals(name, budget, n_recent, mib):
    wl = W.WORKLOADS[name]
    b = bench.step_bytes(wl, budget, n_recent, "carry")
    assert b["total"] == b["select"] + b["draft"] + b["verify"]
    assert b["total"] / MIB == pytest.approx(mib, abs=0.5 if mib > 1 else 0.05)


def test_full_budget_selects_nothing():
    wl = W.WORKLOADS["l8b_16k_b8"]
    assert bench.step_bytes(wl, wl.t_ctx, 0, "carry")["select"] == 0


def test_self_mode_reads_the_prefix_once_more():
    wl = W.WORKLOADS["l8b_16k_b8"]
    carry = bench.step_bytes(wl, 512, 128, "carry")
    own = bench.step_bytes(wl, 512, 128, "self")
    assert own["select"] - carry["select"] == wl.t_ctx * wl.head_dim * 2 * wl.batch * wl.h_kv


def test_stack_totals_with_and_without_the_views_per_pass():
    wl = W.WORKLOADS["l8b_32L_16k_b16"]
    once = bench.step_bytes(wl, wl.budget, wl.n_recent, "carry")["total"] * wl.layers
    assert once / 1e9 == pytest.approx(52.5, abs=0.05)
    assert (once + bench.view_rereads(wl)) / 1e9 == pytest.approx(56.8, abs=0.05)
