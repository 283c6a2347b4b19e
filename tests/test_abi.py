"""Host-side checks of the C ABI (no GPU): the library builds and loads, exports every
entry point include/budgetdraft.h declares, and rejects bad arguments before any
launch.  Only validation paths are exercised: no pointer is dereferenced."""

import ctypes
import os
import re

import pytest

import paper_2606_00144_gb300 as bd
from paper_2606_00144_gb300 import binding

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "budgetdraft.h")

BD_OK, INVALID, UNSUPPORTED, MISALIGNED, WORKSPACE, CUDA_ERR, TIMEOUT = 0, -1, -2, -3, -4, -5, -6
A = 0x10000          # a fake, 16-byte aligned address: validation never dereferences it


@pytest.fixture(scope="module")
def lib():
    bd.build()
    return bd.library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bd_[a-z_]+)\s*\(", text)))


def test_header_declares_the_four_hot_path_calls():
    names = declared_functions()
    for n in ("bd_select_budget", "bd_draft_attn", "bd_verify_attn", "bd_combine"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert sorted(binding.exported_symbols()) == declared_functions()


def test_strerror(lib):
    for code in (BD_OK, INVALID, UNSUPPORTED, MISALIGNED, WORKSPACE, CUDA_ERR, TIMEOUT):
        assert bd.bd_strerror(code) not in ("", "unknown status")
    assert bd.bd_strerror(12345) == "unknown status"


def shape(**kw):
    base = dict(batch=2, h_q=8, h_kv=2, head_dim=128, t_ctx=100, t_cap=110)
    base.update(kw)
    return bd.make_shape(**base)


def verify(lib, s, q=A, n_q=6, k=A, v=A, o=A, lse=A, ws=A, nbytes=1 << 20):
    return lib.bd_verify_attn(ctypes.byref(s) if s is not None else None, q, n_q, k, v, o, lse, ws, nbytes, None)


def draft(lib, s, q=A, k=A, v=A, idx=A, cnt=A, budget=32, j=0, o=A, lse=A, ws=A, nbytes=1 << 20, flags=0):
    return lib.bd_draft_attn(ctypes.byref(s), q, k, v, idx, cnt, budget, j, flags, o, lse, ws, nbytes, None)


def select(lib, s, k=A, qw=A, lse=A, window=32, budget=40, sink=4, recent=8, chunk=1, idx=A, cnt=A, ws=A,
           nbytes=1 << 20, flags=0):
    return lib.bd_select_budget(ctypes.byref(s), k, qw, lse, window, budget, sink, recent, chunk, flags, idx, cnt,
                                ws, nbytes, None)


def test_verify_validation(lib):
    assert verify(lib, None) == INVALID
    assert verify(lib, shape(head_dim=96)) == UNSUPPORTED
    assert verify(lib, shape(h_q=6, h_kv=4)) == INVALID             # h_q % h_kv != 0
    assert verify(lib, shape(t_cap=50)) == INVALID                    # t_cap < t_ctx
    assert verify(lib, shape(), q=0) == INVALID
    assert verify(lib, shape(), k=A + 8) == MISALIGNED
    assert verify(lib, shape(), o=A + 2) == MISALIGNED
    assert verify(lib, shape(), n_q=0) == INVALID
    assert verify(lib, shape(), n_q=11) == INVALID                    # t_ctx + n_q > t_cap
    assert verify(lib, shape(), n_q=2**31 - 1) == INVALID             # the sum does not wrap
    assert verify(lib, shape(), o=0, lse=0) == INVALID                # nothing to write
    assert verify(lib, shape(t_cap=400), n_q=193) == UNSUPPORTED      # 4 * 193 rows > 768 with V
    assert verify(lib, shape(t_cap=200), n_q=33, o=0) == UNSUPPORTED  # 4 * 33 rows > 128, lse only


def test_draft_validation(lib):
    assert draft(lib, shape(), idx=0) == INVALID
    assert draft(lib, shape(), cnt=A + 2) == MISALIGNED
    assert draft(lib, shape(), j=-1) == INVALID
    assert draft(lib, shape(), j=10) == INVALID                       # t_ctx + j >= t_cap
    assert draft(lib, shape(), j=2**31 - 1) == INVALID                # the sum does not wrap
    assert draft(lib, shape(), budget=0) == INVALID
    assert draft(lib, shape(h_q=34, h_kv=2)) == UNSUPPORTED           # group of 17 > 16
    assert draft(lib, shape(h_q=18, h_kv=2)) != UNSUPPORTED           # group of 9: two query tiles
    assert draft(lib, shape(), flags=6) == INVALID                    # unknown flag bits


def test_draft_view_beyond_shared_memory_is_unsupported(lib):
    """The row table of a CTA's slice lives in shared memory: a view of a million entries
    cannot be planned (size 0, BD_ERR_UNSUPPORTED), a 4K view can."""
    s = shape(t_ctx=2_000_000, t_cap=2_000_010)
    assert lib.bd_workspace_size(ctypes.byref(s), binding.BD_OP_DRAFT, 1_000_000, 1) == 0
    assert lib.bd_workspace_size(ctypes.byref(s), binding.BD_OP_DRAFT, 4096, 1) > 0
    assert draft(lib, s, budget=1_000_000) == UNSUPPORTED


def test_select_validation(lib):
    assert select(lib, shape(), window=0) == INVALID
    assert select(lib, shape(), window=101) == INVALID                # window > t_ctx
    assert select(lib, shape(), budget=10, sink=4, recent=8) == INVALID   # sink + recent > budget
    assert select(lib, shape(), budget=10, sink=2**31 - 1, recent=2**31 - 1) == INVALID   # no wrap
    assert select(lib, shape(), chunk=0) == INVALID
    assert select(lib, shape(), flags=2) == INVALID                   # unknown flag bits
    assert select(lib, shape(), sink=-1) == INVALID
    assert select(lib, shape(), lse=A + 1) == MISALIGNED
    assert select(lib, shape(h_q=16, h_kv=1), window=32) == UNSUPPORTED  # 512 window rows > 256
    assert select(lib, shape(h_q=16, h_kv=2), window=32, lse=None) == UNSUPPORTED   # self mode: 256 rows > 128
    assert select(lib, shape(), qw=0) == INVALID


def test_combine_validation(lib):
    f = lib.bd_combine
    assert f(A, A, 0, 4, 128, A, A, None) == INVALID
    assert f(A, A, 2, -1, 128, A, A, None) == INVALID
    assert f(A, A, 2, 4, 32, A, A, None) == UNSUPPORTED
    assert f(A, A, 12289, 4, 128, A, A, None) == UNSUPPORTED            # weights beyond 48 KB of smem
    assert f(A, A, 2, 0, 128, A, A, None) == BD_OK                     # empty: no-op
    assert f(A + 4, A, 2, 4, 128, A, A, None) == MISALIGNED
    assert f(A, A, 2, 4, 128, 0, A, None) == INVALID


def test_workspace_status_null(lib):
    assert lib.bd_workspace_status(None, None) == INVALID


def test_product_path_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError):
        binding.library()


def test_argmax_validation(lib):
    f = lib.bd_argmax
    assert f(A, 3, 4, 100, A, None) == INVALID                         # unknown dtype
    assert f(A, binding.BD_DTYPE_BF16, -1, 100, A, None) == INVALID
    assert f(A, binding.BD_DTYPE_BF16, 4, 0, A, None) == INVALID
    assert f(A, binding.BD_DTYPE_BF16, 0, 100, A, None) == BD_OK         # empty: no-op
    assert f(A, binding.BD_DTYPE_BF16, 70000, 100, A, None) == UNSUPPORTED
    assert f(A, binding.BD_DTYPE_BF16, 4, (1 << 30) + 1, A, None) == UNSUPPORTED   # indices past 2^31
    assert f(A + 1, binding.BD_DTYPE_BF16, 4, 100, A, None) == MISALIGNED
    assert f(A + 2, binding.BD_DTYPE_F32, 4, 100, A, None) == MISALIGNED
    assert f(A, binding.BD_DTYPE_F32, 4, 100, A + 2, None) == MISALIGNED
    assert f(A, binding.BD_DTYPE_F32, 4, 100, None, None) == INVALID
    assert f(None, binding.BD_DTYPE_F32, 4, 100, A, None) == INVALID


def test_accept_validation(lib):
    f = lib.bd_accept
    assert f(-1, 5, A, A, A, A, None) == INVALID
    assert f(8, -1, A, A, A, A, None) == INVALID
    assert f(0, 5, None, None, None, None, None) == BD_OK               # empty: no-op
    assert f(8, 5, A, A, None, None, None) == INVALID                    # nothing to write
    assert f(8, 5, None, A, A, A, None) == INVALID                       # drafts needed when gamma > 0
    assert f(8, 5, A, None, A, A, None) == INVALID
    assert f(8, 5, A, A, A + 2, A, None) == MISALIGNED
    assert f(8, 5, A, A, A, A + 1, None) == MISALIGNED


def test_advance_validation(lib):
    def adv(s, window=32, n_q=6, n_acc=A, qv=A, lv=A, qw=A, lw=A, idx=A, cnt=A, cap=64, out=A):
        return lib.bd_advance(ctypes.byref(s), window, n_q, n_acc, qv, lv, qw, lw, idx, cnt, cap, out, None)
    assert adv(shape(), window=0) == INVALID
    assert adv(shape(), window=101) == INVALID                          # window > t_ctx
    assert adv(shape(), n_q=11) == INVALID                              # t_ctx + n_q > t_cap
    assert adv(shape(), n_q=2**31 - 1) == INVALID                       # the sum does not wrap
    assert adv(shape(), lv=None) == INVALID                             # lse ring needs both sides
    assert adv(shape(), cnt=None) == INVALID                            # view needs idx and count
    assert adv(shape(), cap=0) == INVALID
    assert adv(shape(), n_acc=None) == INVALID
    assert adv(shape(), qw=A + 8) == MISALIGNED
    assert adv(shape(), out=A + 2) == MISALIGNED
    assert adv(shape(head_dim=96)) == UNSUPPORTED


def test_write_block_rows_validation(lib):
    f = lib.bd_write_block_rows
    assert f(ctypes.byref(shape()), 0, A, A, A, A, None) == INVALID
    assert f(ctypes.byref(shape()), 11, A, A, A, A, None) == INVALID      # t_ctx + n_rows > t_cap
    assert f(ctypes.byref(shape()), 2**31 - 1, A, A, A, A, None) == INVALID   # the sum does not wrap
    assert f(ctypes.byref(shape()), 6, A + 8, A, A, A, None) == MISALIGNED
    assert f(ctypes.byref(shape()), 6, A, A, None, A, None) == INVALID
    assert f(ctypes.byref(shape(head_dim=96)), 6, A, A, A, A, None) == UNSUPPORTED


def test_seq_lens_pointer_is_checked(lib):
    s = shape()
    s.seq_lens = A + 2
    assert verify(lib, s) == MISALIGNED
    s.seq_lens = A
    assert verify(lib, s, n_q=0) == INVALID            # the other checks still run


def test_plain_c_consumer(lib, tmp_path):
    # the header compiles as C and the library links and answers from a C program
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    here = os.path.dirname(__file__)
    exe = tmp_path / "consumer"
    lib_dir = os.path.dirname(bd.LIB_PATH)
    subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER),
                    os.path.join(here, "c_abi_consumer.c"), "-o", str(exe), "-L", lib_dir, "-lbudgetdraft",
                    f"-Wl,-rpath,{lib_dir}"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    assert out[0] == "workspace_size 0"
    assert out[1] == f"verify {UNSUPPORTED}"
    assert out[2] == f"argmax {INVALID}"
    assert out[3] == f"accept_empty {BD_OK}"
    assert out[4] == "strerror " + bd.bd_strerror(MISALIGNED)


def test_check_wait_timeout_validation(lib):
    f = lib.bd_check_wait_timeout
    assert f(None, 1024, 1000, None) == INVALID
    assert f(A, 16, 1000, None) == WORKSPACE
    assert f(A, 1024, 0, None) == INVALID
    assert f(A, 1024, 3000000, None) == INVALID
    assert f(A + 4, 1024, 1000, None) == MISALIGNED


def test_seq_lens_unit_limit(lib):
    s = shape(batch=513, h_q=64, h_kv=8)          # 4104 units: beyond the 4096 the tables allow
    s.seq_lens = A
    assert verify(lib, s) == UNSUPPORTED
    s = shape(batch=129, h_q=64, h_kv=8)          # 1032 units: within them
    s.seq_lens = A
    assert verify(lib, s) != UNSUPPORTED
