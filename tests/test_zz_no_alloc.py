"""The allocation-free group selection (htam_select_groups_static) against
htam_query's own group selection, through the C ABI (GPU).

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

pytestmark = pytest.mark.gpu

GAP = 1e-3
TOL = {torch.bfloat16: (2e-2, 1e-4), torch.float32: (1e-5, 1e-7)}


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
    return htam.Memory(x, gid, g), centres


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


def _agree(gi, gs, ref_gi, ref_gs, dtype):
    """Same ids except swaps inside near-ties; scores within the parity tolerance."""
    rtol, atol = TOL[dtype]
    gi, gs, ref_gi, ref_gs = (t.cpu().numpy() for t in (gi, gs, ref_gi, ref_gs))
    for b in range(gi.shape[0]):
        if not np.array_equal(gi[b], ref_gi[b]):
            gaps = np.abs(np.diff(ref_gs[b]))
            assert set(gi[b]) == set(ref_gi[b]) and (gaps < GAP).any(), f"query {b}: {gi[b]} vs {ref_gi[b]}"
        ok = np.isneginf(ref_gs[b]) == np.isneginf(gs[b])
        fin = ~np.isneginf(ref_gs[b])
        ok[fin] &= np.abs(gs[b][fin] - ref_gs[b][fin]) <= rtol * np.abs(ref_gs[b][fin]) + atol
        assert ok.all(), f"query {b}: scores {gs[b]} vs {ref_gs[b]}"


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_static_selection_matches_htam_query_twice(htam, dtype):
    mem, centres = _memory(htam, 40000, 256, 300, dtype, seed=1)
    qa = _queries(centres, 500, dtype, seed=2)
    qb = _queries(centres, 77, dtype, seed=3)   # smaller second call: stale rows from the first stay behind
    kg = 12
    ref_a = mem.query(qa, kg, 4)
    ref_b = mem.query(qb, kg, 4)
    rc_a, gi_a, gs_a = _select_static(htam, mem, qa, kg)
    rc_b, gi_b, gs_b = _select_static(htam, mem, qb, kg)
    torch.cuda.synchronize()
    assert rc_a == htam.HTAM_OK and rc_b == htam.HTAM_OK
    _agree(gi_a, gs_a, ref_a["group_idx"], ref_a["group_score"], dtype)
    _agree(gi_b, gs_b, ref_b["group_idx"], ref_b["group_score"], dtype)


def test_static_selection_pads_and_rejects_oversize(htam):
    gid = torch.tensor([2, 5, 9] * 40, dtype=torch.int32, device="cuda")  # 3 of 20 groups non-empty
    x = torch.randn(gid.numel(), 32, device="cuda")
    mem = htam.Memory((x / x.norm(dim=1, keepdim=True)).contiguous(), gid, 20)
    q = torch.randn(9, 32, device="cuda")
    ref = mem.query(q, 5, 3)
    rc, gi, gs = _select_static(htam, mem, q, 5)
    torch.cuda.synchronize()
    assert rc == htam.HTAM_OK
    assert (gi[:, 3:] == -1).all()
    _agree(gi, gs, ref["group_idx"], ref["group_score"], torch.float32)
    # b * n_groups * 4 bytes above the fixed scratch: rejected, nothing launched.
    big_b = (16 << 20) // (4 * 20) + 1
    qbig = torch.zeros(big_b, 32, device="cuda")
    rc, _, _ = _select_static(htam, mem, qbig, 5)
    assert rc == htam.HTAM_EINVAL
