"""The allocation-free group selection (htam_select_groups_static) through the
C ABI (GPU): against the float64 oracle's stage 1, by the same index and value
rule as every other stage-1 parity test, and against htam_query's own group
selection.

htam_select_groups_static exists for callers that cannot allocate device
memory while they run (a fully pre-reserved memory budget, allocator
callbacks, loops that cannot absorb cudaFree's device-wide synchronisation);
its scratch is a fixed array inside the library.  This file is collected last
so that a failing run stopped at the first failure has already run the rest.
"""
import ctypes

import numpy as np
import pytest
import torch

from parity import check_ranked, close
from paper_2605_29734_gb300.workloads import to_numpy

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def htam():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2605_29734_gb300 import htam as mod

    return mod


def _memory(htam, n, d, g, dtype, seed):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    gid = torch.randint(0, g, (n,), generator=gen, device="cuda", dtype=torch.int64).to(torch.int32)
    centres = torch.randn(g, d, generator=gen, device="cuda")
    x = centres[gid.long()] + 0.3 * torch.randn(n, d, generator=gen, device="cuda")
    x = (x / torch.linalg.vector_norm(x, dim=1, keepdim=True)).to(dtype).contiguous()
    return htam.Memory(x, gid, g), centres, x, gid


def _queries(centres, b, dtype, seed):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    pick = torch.randint(0, centres.shape[0], (b,), generator=gen, device="cuda")
    x = centres[pick] + 0.3 * torch.randn(b, centres.shape[1], generator=gen, device="cuda")
    return (x / torch.linalg.vector_norm(x, dim=1, keepdim=True)).to(dtype).contiguous()


def _select_static(htam, mem, q, kg):
    b = q.shape[0]
    gi = torch.full((b, kg), -7, dtype=torch.int32, device="cuda")
    gs = torch.full((b, kg), 7.0, dtype=torch.float32, device="cuda")
    rc = htam.lib().htam_select_groups_static(mem.handle, ctypes.c_void_p(q.data_ptr()), b, kg,
                                              ctypes.c_void_p(gi.data_ptr()), ctypes.c_void_p(gs.data_ptr()),
                                              ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return rc, gi, gs


def _against_oracle(gi, gs, x, gid, g, q, kg, dtype):
    """Stage 1 of the oracle (float64 keys and scores) with k_groups + 1
    ranked, so the k-th / (k+1)-th gap decides how strict the id check is."""
    import oracle

    cent, counts = oracle.centroids(to_numpy(x), to_numpy(gid), g)
    qn = to_numpy(q)
    qf = (qn.astype(np.uint32) << 16).view(np.float32).astype(np.float64) if qn.dtype == np.uint16 else \
        qn.astype(np.float64)
    ref_gi, ref_gs = oracle.stage1(qn, cent, counts, min(kg + 1, g))
    if ref_gi.shape[1] == kg:
        ref_gi = np.concatenate([ref_gi, -np.ones((len(ref_gi), 1), np.int32)], axis=1)
        ref_gs = np.concatenate([ref_gs, np.full((len(ref_gs), 1), -np.inf)], axis=1)
    gi, gs = gi.cpu().numpy(), gs.cpu().numpy()
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    problems = []
    for b in range(gi.shape[0]):
        problems += check_ranked(f"query {b} groups", gi[b], gs[b], ref_gi[b], ref_gs[b], kg,
                                 lambda gg, b=b: float(cent[gg] @ qf[b]), dt)
    return problems


def _against_query(gi, gs, ref_gi, ref_gs, dtype):
    """Same ids as htam_query's stage 1 wherever its adjacent scores differ
    by more than the index gap; scores within the parity tolerance."""
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    gi, gs, ref_gi, ref_gs = (t.cpu().numpy() for t in (gi, gs, ref_gi, ref_gs))
    problems = []
    for b in range(gi.shape[0]):
        for i in range(gi.shape[1]):
            if ref_gi[b, i] < 0:  # padding: -1 / -inf on both sides
                if gi[b, i] != -1 or not np.isneginf(gs[b, i]):
                    problems.append(f"query {b} slot {i}: padding {gi[b, i]} {gs[b, i]}")
                continue
            clear_above = i == 0 or ref_gs[b, i - 1] - ref_gs[b, i] > 1e-3
            clear_below = i + 1 == gi.shape[1] or ref_gi[b, i + 1] < 0 or ref_gs[b, i] - ref_gs[b, i + 1] > 1e-3
            if clear_above and clear_below and gi[b, i] != ref_gi[b, i]:
                problems.append(f"query {b} slot {i}: {gi[b, i]} vs htam_query {ref_gi[b, i]}")
            if not close(gs[b, i], ref_gs[b, i], dt):
                problems.append(f"query {b} slot {i}: score {gs[b, i]} vs htam_query {ref_gs[b, i]}")
    return problems


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_static_selection_matches_oracle_and_htam_query_twice(htam, dtype):
    """Two calls in a row (the second smaller, so rows of the first stay
    behind in the shared array), each against the oracle and htam_query."""
    g, kg = 300, 12
    mem, centres, x, gid = _memory(htam, 40000, 256, g, dtype, seed=1)
    qa = _queries(centres, 500, dtype, seed=2)
    qb = _queries(centres, 77, dtype, seed=3)
    ref_a = mem.query(qa, kg, 4)
    ref_b = mem.query(qb, kg, 4)
    rc_a, gi_a, gs_a = _select_static(htam, mem, qa, kg)
    rc_b, gi_b, gs_b = _select_static(htam, mem, qb, kg)
    torch.cuda.synchronize()
    assert rc_a == htam.HTAM_OK and rc_b == htam.HTAM_OK
    problems = _against_oracle(gi_a, gs_a, x, gid, g, qa, kg, dtype)
    problems += _against_oracle(gi_b, gs_b, x, gid, g, qb, kg, dtype)
    problems += _against_query(gi_a, gs_a, ref_a["group_idx"], ref_a["group_score"], dtype)
    problems += _against_query(gi_b, gs_b, ref_b["group_idx"], ref_b["group_score"], dtype)
    assert not problems, "\n".join(problems[:20])


def test_static_selection_allocates_nothing(htam):
    """After the first call (which looks up the array's device address), calls
    of several sizes leave the device's free memory exactly where it was."""
    mem, centres, _, _ = _memory(htam, 20000, 128, 200, torch.bfloat16, seed=4)
    qs = [_queries(centres, b, torch.bfloat16, seed=10 + b) for b in (1, 300, 4000, 20000)]
    rc, _, _ = _select_static(htam, mem, qs[0], 8)
    torch.cuda.synchronize()
    assert rc == htam.HTAM_OK
    outs = [(torch.empty(q.shape[0], 8, dtype=torch.int32, device="cuda"),
             torch.empty(q.shape[0], 8, dtype=torch.float32, device="cuda")) for q in qs]
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info()
    for _ in range(2):
        for q, (gi, gs) in zip(qs, outs):
            rc = htam.lib().htam_select_groups_static(
                mem.handle, ctypes.c_void_p(q.data_ptr()), q.shape[0], 8, ctypes.c_void_p(gi.data_ptr()),
                ctypes.c_void_p(gs.data_ptr()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
            assert rc == htam.HTAM_OK
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert free_after == free_before


def test_static_selection_pads_and_rejects_oversize(htam):
    gid = torch.tensor([2, 5, 9] * 40, dtype=torch.int32, device="cuda")  # 3 of 20 groups non-empty
    x = torch.randn(gid.numel(), 32, device="cuda")
    x = (x / x.norm(dim=1, keepdim=True)).contiguous()
    mem = htam.Memory(x, gid, 20)
    q = torch.randn(9, 32, device="cuda")
    q = (q / q.norm(dim=1, keepdim=True)).contiguous()
    ref = mem.query(q, 5, 3)
    rc, gi, gs = _select_static(htam, mem, q, 5)
    torch.cuda.synchronize()
    assert rc == htam.HTAM_OK
    assert (gi[:, 3:] == -1).all() and torch.isneginf(gs[:, 3:]).all()
    problems = _against_oracle(gi, gs, x, gid, 20, q, 5, torch.float32)
    problems += _against_query(gi, gs, ref["group_idx"], ref["group_score"], torch.float32)
    assert not problems, "\n".join(problems[:20])
    # b * n_groups * 4 bytes above the fixed scratch: rejected, nothing launched.
    big_b = (16 << 20) // (4 * 20) + 1
    qbig = torch.zeros(big_b, 32, device="cuda")
    rc, _, _ = _select_static(htam, mem, qbig, 5)
    assert rc == htam.HTAM_EINVAL


def test_static_selection_more_query_tiles_than_a_grid_row(htam):
    """With one group, 2,100,000 queries fit the fixed scratch (8.4 MB) and
    take 65,625 32-query tiles: more than a launch's grid.y allows, so the
    query tiles must sit on grid.x.  Every query selects the one group; the
    scores are checked against the oracle's on a sample."""
    import oracle

    mem, centres, x, gid = _memory(htam, 500, 32, 1, torch.float32, seed=5)
    b = 2_100_000
    q = torch.randn(b, 32, generator=torch.Generator(device="cuda").manual_seed(6), device="cuda")
    q = (q / torch.linalg.vector_norm(q, dim=1, keepdim=True)).contiguous()
    rc, gi, gs = _select_static(htam, mem, q, 1)
    torch.cuda.synchronize()
    assert rc == htam.HTAM_OK
    assert (gi == 0).all()
    cent, _ = oracle.centroids(to_numpy(x), to_numpy(gid), 1)
    rows = np.linspace(0, b - 1, 4096).astype(int)
    want = q[rows].double().cpu().numpy() @ cent[0]
    got = gs[rows, 0].cpu().numpy()
    assert all(close(gv, wv, "f32") for gv, wv in zip(got, want))
