"""Register and spill budget of the kernels, from ptxas (-Xptxas -v) with the library's own
build flags: the instances that one step of each synthetic workload runs (d 64 / 128, GQA
group 4, a 32-row window, gamma 5) must not spill to local memory, and no instance may spill
more than a few words.  Compiles on the CPU; skipped where nvcc is missing."""

import concurrent.futures
import importlib
import os
import re
import shutil
import subprocess

import pytest

B = importlib.import_module("paper_2606_00144_gb300.build")   # the module (the package re-exports build())

ENTRY = re.compile(r"Compiling entry function '(\w+)' for '(\w+)'")
SPILL = re.compile(r"(\d+) bytes stack frame, (\d+) bytes spill stores, (\d+) bytes spill loads")
REGS = re.compile(r"Used (\d+) registers")

# mangled-name patterns of the instances the workloads' steps launch
NO_SPILL = {
    "score kernel, uniform lengths": r"_ZN2bd12score_kernelILi\d+ELi\d+ELi\d+ELb0E",
    "window-LSE kernel, uniform lengths": r"_ZN2bd17window_lse_kernelILi\d+ELb0E",
    "register top-B kernels": r"_ZN2bd(16topk_rows_kernel|22topk_rows_chunk_kernel)ILi\d+E",
    "draft kernel, group 4": r"_ZN2bd12draft_kernelILi(64|128)ELi4E",
    "verify kernel, 24 rows with V": r"_ZN2bd13verify_kernelILi(64|128)ELi3ELi1ELb1ELb0E",
}
MAX_SPILL_STORE_BYTES = 32   # eight words of local memory


@pytest.fixture(scope="module")
def resources(tmp_path_factory):
    try:
        nvcc = B.nvcc_path()
    except RuntimeError:
        pytest.skip("nvcc not available")
    out = tmp_path_factory.mktemp("ptxas")

    def one(src):
        cmd = [nvcc, *B.FLAGS, "-Xptxas", "-v", "-c", os.path.join(B.CSRC, src), "-o", str(out / (src + ".o"))]
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stderr[-2000:]
        return r.stdout + r.stderr

    with concurrent.futures.ThreadPoolExecutor(max_workers=len(B.SOURCES)) as ex:
        logs = list(ex.map(one, B.SOURCES))
    kernels = {}
    for log in logs:
        name = None
        for line in log.splitlines():
            m = ENTRY.search(line)
            if m:
                name = m.group(1)
                kernels[name] = dict(arch=m.group(2), spill=0, reload=0, regs=None)
                continue
            if name is None:
                continue
            m = SPILL.search(line)
            if m:
                kernels[name]["spill"] = int(m.group(2))
                kernels[name]["reload"] = int(m.group(3))
            m = REGS.search(line)
            if m:
                kernels[name]["regs"] = int(m.group(1))
    shutil.rmtree(out, ignore_errors=True)
    return kernels


def test_every_kernel_is_built_for_sm_103a(resources):
    assert resources, "ptxas reported no kernels"
    assert {k["arch"] for k in resources.values()} == {"sm_103a"}
    assert all(k["regs"] is not None and k["regs"] <= 255 for k in resources.values())


@pytest.mark.parametrize("what", sorted(NO_SPILL))
def test_workload_instances_do_not_spill(resources, what):
    pat = re.compile(NO_SPILL[what])
    hits = {n: k for n, k in resources.items() if pat.match(n)}
    assert hits, f"no instance matches {what}"
    spilled = {n: (k["spill"], k["reload"]) for n, k in hits.items() if k["spill"] or k["reload"]}
    assert not spilled, f"{what}: {spilled}"


def test_no_instance_spills_more_than_a_few_words(resources):
    big = {n: k["spill"] for n, k in resources.items() if k["spill"] > MAX_SPILL_STORE_BYTES}
    assert not big, big
