"""Parity of the greedy acceptance calls (Eq. accept; Algorithm 2, accept and bonus token)
with the oracle: bd_argmax over vocabulary rows and bd_accept over token blocks.  Both are
integer results, so the bar is bit-exact."""

import numpy as np
import pytest
import torch

import oracle
import paper_2606_00144_gb300 as bd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    bd.build()
    bd.library()


def logits_rows(rows, vocab, dtype, seed, specials=True):
    """Seeded N(0, 1) logits; with `specials`, some rows carry planted ties, NaN, -inf and
    signed zeros (the cases the arg max rule has to order)."""
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(rows, vocab, generator=g).to(dtype)
    if specials and rows >= 6 and vocab >= 4:
        top = x.float().max(dim=1).values
        x[0, vocab - 1] = top[0] + 1                      # maximum in the last element
        x[0, vocab // 2] = top[0] + 1                     # ... tied with a lower id
        x[1, :] = float("nan")                            # nothing comparable -> 0
        x[2, :] = float("-inf")                           # all -inf -> the first id
        x[2, 0] = float("nan")                            # ... but never a NaN
        x[3, :] = -1.0
        x[3, 2] = -0.0
        x[3, 1] = 0.0                                     # -0 == +0: the lower id wins
        x[4, 0] = float("nan")
        x[4, 1:] = float("-inf")                          # first comparable element
        x[5, :] = float("inf")                            # all +inf -> 0
    return x


def check_argmax(x):
    ids = torch.empty(x.shape[0], dtype=torch.int32, device="cuda")
    xd = x.cuda()
    bd.bd_argmax(xd, ids)
    torch.cuda.synchronize()
    ref = oracle.greedy_argmax(x.float().numpy() if x.dtype == torch.bfloat16 else x.numpy())
    got = ids.cpu().numpy()
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, f"rows {bad[:8]}: got {got[bad[:8]]} want {ref[bad[:8]]}"


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("rows,vocab", [(1, 1), (6, 7), (8, 4095), (48, 32000), (40, 128256), (300, 1000),
                                        (7, 128257)])
def test_argmax_matches_oracle(rows, vocab, dtype):
    check_argmax(logits_rows(rows, vocab, dtype, seed=rows * 7919 + vocab))


def test_argmax_dense_ties_bf16():
    # few distinct values: nearly every row has many tied maxima
    g = torch.Generator().manual_seed(5)
    x = torch.randint(-4, 4, (64, 50000), generator=g).to(torch.bfloat16)
    check_argmax(x)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_argmax_scattered_nan_and_inf(dtype):
    # NaN at 30% of the positions (whole 16-byte vectors of NaN included), +-inf sprinkled
    g = torch.Generator().manual_seed(7)
    x = torch.randint(-3, 3, (96, 20000), generator=g).to(dtype)
    x[torch.rand(x.shape, generator=g) < 0.3] = float("nan")
    x[torch.rand(x.shape, generator=g) < 0.01] = float("-inf")
    x[10:20] = float("-inf")
    x[10:20][torch.rand(10, 20000, generator=g) < 0.5] = float("nan")
    x[20:22, 12345] = float("inf")
    check_argmax(x)


def test_argmax_unaligned_row_starts():
    # a view starting one element into a buffer: every row begins off the 16-byte phase
    g = torch.Generator().manual_seed(6)
    base = torch.randn(12 * 9999 + 1, generator=g).to(torch.bfloat16).cuda()
    x = base[1:].view(12, 9999)
    ids = torch.empty(12, dtype=torch.int32, device="cuda")
    bd.bd_argmax(x, ids)
    torch.cuda.synchronize()
    assert ids.cpu().numpy().tolist() == oracle.greedy_argmax(x.float().cpu().numpy()).tolist()


def token_blocks(batch, gamma, seed):
    """Drafter / verifier tokens with every agreement length 0..gamma represented."""
    rng = np.random.default_rng(seed)
    d = rng.integers(0, 128256, size=(batch, gamma)).astype(np.int32)
    v = rng.integers(0, 128256, size=(batch, gamma + 1)).astype(np.int32)
    k = rng.integers(0, gamma + 1, size=batch)
    for b in range(batch):
        v[b, :k[b]] = d[b, :k[b]]
        if k[b] + 1 < gamma and rng.random() < 0.5:
            v[b, k[b] + 1:gamma] = d[b, k[b] + 1:gamma]    # agreement after the first mismatch
    return d, v


@pytest.mark.parametrize("batch,gamma", [(1, 0), (1, 1), (8, 5), (33, 8), (1000, 5), (4, 31)])
def test_accept_matches_oracle(batch, gamma):
    d, v = token_blocks(batch, gamma, seed=batch * 31 + gamma)
    n = torch.full((batch,), -7, dtype=torch.int32, device="cuda")
    emit = torch.full((batch, gamma + 1), -7, dtype=torch.int32, device="cuda")
    dd = torch.from_numpy(np.ascontiguousarray(d.T)).cuda() if gamma > 0 else None   # pass-major
    bd.bd_accept(dd, torch.from_numpy(v).cuda(), n, emit)
    torch.cuda.synchronize()
    n_ref, emit_ref = oracle.accept_greedy(d, v)
    assert n.cpu().numpy().tolist() == n_ref.tolist()
    assert emit.cpu().numpy().tolist() == emit_ref.tolist()


def test_accept_from_logits_pipeline():
    # a whole greedy accept: drafter argmax per pass, verifier argmax over the block, accept
    batch, gamma, vocab = 8, 5, 128256
    g = torch.Generator().manual_seed(11)
    draft_logits = torch.randn(gamma, batch, vocab, generator=g).to(torch.bfloat16)
    verify_logits = torch.randn(batch, gamma + 1, vocab, generator=g).to(torch.bfloat16)
    # plant agreement: copy the drafter's rows into the verifier's for a prefix of each sequence
    for b in range(batch):
        for i in range(b % (gamma + 1)):
            verify_logits[b, i] = draft_logits[i, b]
    dl, vl = draft_logits.cuda(), verify_logits.cuda()
    d_ids = torch.empty(gamma, batch, dtype=torch.int32, device="cuda")
    v_ids = torch.empty(batch, gamma + 1, dtype=torch.int32, device="cuda")
    for j in range(gamma):
        bd.bd_argmax(dl[j], d_ids[j])
    bd.bd_argmax(vl.view(batch * (gamma + 1), vocab), v_ids.view(-1))
    n = torch.empty(batch, dtype=torch.int32, device="cuda")
    emit = torch.empty(batch, gamma + 1, dtype=torch.int32, device="cuda")
    bd.bd_accept(d_ids, v_ids, n, emit)
    torch.cuda.synchronize()
    d_ref = oracle.greedy_argmax(draft_logits.float().numpy().reshape(-1, vocab)).reshape(gamma, batch).T
    v_ref = oracle.greedy_argmax(verify_logits.float().numpy().reshape(-1, vocab)).reshape(batch, gamma + 1)
    n_ref, emit_ref = oracle.accept_greedy(d_ref, v_ref)
    assert n.cpu().numpy().tolist() == n_ref.tolist()
    assert emit.cpu().numpy().tolist() == emit_ref.tolist()
    assert n_ref.tolist() != [0] * batch          # the planted prefixes were seen
