"""Parity of the CUDA lookup with the float64 oracle, through the C ABI (GPU)."""
import numpy as np
import pytest
import torch

from parity import compare_lookup, edge_score_tol
from paper_2605_29734_gb300 import workloads
from paper_2605_29734_gb300.workloads import to_numpy

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def htam():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2605_29734_gb300 import htam as mod

    return mod


DEV = "cuda"


def _unit(x):
    return x / torch.linalg.vector_norm(x, dim=1, keepdim=True)


def _rand_memory(n, d, g, dtype, seed, clustered=True, gid=None):
    gen = torch.Generator(device=DEV).manual_seed(seed)
    if gid is None:
        gid = torch.randint(0, g, (n,), generator=gen, device=DEV, dtype=torch.int64).to(torch.int32)
    if clustered:
        centres = torch.randn(g, d, generator=gen, device=DEV)
        x = centres[gid.long()] + 0.3 * torch.randn(n, d, generator=gen, device=DEV)
    else:
        centres = None
        x = torch.randn(n, d, generator=gen, device=DEV)
    return _unit(x).to(dtype).contiguous(), gid.contiguous(), centres


def _rand_queries(b, d, dtype, seed, centres=None):
    gen = torch.Generator(device=DEV).manual_seed(seed + 7)
    if centres is not None:
        pick = torch.randint(0, centres.shape[0], (b,), generator=gen, device=DEV)
        x = centres[pick] + 0.3 * torch.randn(b, d, generator=gen, device=DEV)
    else:
        x = torch.randn(b, d, generator=gen, device=DEV)
    return _unit(x).to(dtype).contiguous()


def _check(htam, mem, entries, gid, g, queries, kg, ke, tau=1.0, eps=0.0, rows=None, **kw):
    out = mem.query(queries, kg, ke, tau=tau, epsilon=eps)
    torch.cuda.synchronize()
    dt = "bf16" if queries.dtype == torch.bfloat16 else "f32"
    problems = compare_lookup(out, to_numpy(entries), to_numpy(gid), g, to_numpy(queries), kg, ke, tau, eps,
                              dt, rows=rows, **kw)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK
    return out


# ------------------------------------------------------------- workload sizes

@pytest.mark.parametrize("tau,eps", [(1.0, 0.0), (0.05, 0.0), (1.0, 0.1), (0.5, 1.0)])
def test_tiny_fp32_workload(htam, tau, eps):
    w = workloads.WORKLOADS["tiny_f32_1k"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    q = workloads.make_queries(w, gid, centres, seed=0)
    mem = htam.Memory(entries, gid, w.g)
    _check(htam, mem, entries, gid, w.g, q, w.k_groups, w.k_entries, tau, eps)


def test_zipf_65k_workload(htam):
    w = workloads.WORKLOADS["zipf_bf16_65k"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    q = workloads.make_queries(w, gid, centres, seed=0)
    mem = htam.Memory(entries, gid, w.g)
    _check(htam, mem, entries, gid, w.g, q, w.k_groups, w.k_entries)


def _bench_batches(w, gid, centres, n=4):
    """The query batches the benchmark cycles over (seed 0, rank 0)."""
    return [workloads.make_queries(w, gid, centres, seed=0, stream=4 + 10 * i) for i in range(n)]


def test_zipf_1m_workload_every_bench_batch(htam):
    """Full size (1,048,576 entries, 1,024 Zipf groups, d = 1,024), every
    query of every batch the benchmark times (4 x 4,096), in the benchmark's
    launch configuration: stage 1 against the oracle's float64 group scores
    (Eq. 12's restriction starts from these groups), stage 2 given the GPU's
    groups (Eq. 13's pick, Eq. 11's weights and lse)."""
    import oracle

    w = workloads.WORKLOADS["zipf_bf16_1m"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    mem = htam.Memory(entries, gid, w.g)
    entries_np, gid_np = to_numpy(entries), to_numpy(gid)
    cent, counts = oracle.centroids(entries_np, gid_np, w.g)
    for i, q in enumerate(_bench_batches(w, gid, centres)):
        out = mem.query(q, w.k_groups, w.k_entries)
        torch.cuda.synchronize()
        problems = compare_lookup(out, entries_np, gid_np, w.g, to_numpy(q), w.k_groups, w.k_entries, 1.0, 0.0,
                                  "bf16", centroid=cent, counts=counts)
        assert not problems, f"batch {i}:\n" + "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


def test_uniform_4m_workload_every_bench_batch(htam):
    """The largest memory (4,194,304 x 4,096 bf16, 32 GiB of keys): every
    query of every batch the benchmark times (4 x 64); the oracle's group
    keys are accumulated from the host copy once.  The flat scan on the same
    memory is checked on a sample of the first batch."""
    import oracle

    w = workloads.WORKLOADS["uniform_bf16_4m"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    mem = htam.Memory(entries, gid, w.g)
    batches = _bench_batches(w, gid, centres)
    outs = []
    for q in batches:
        outs.append({k: v.clone() for k, v in mem.query(q, w.k_groups, w.k_entries).items()})
    flat = mem.query_flat(batches[0], w.k_entries)
    torch.cuda.synchronize()
    entries_np = to_numpy(entries)
    gid_np = to_numpy(gid)
    del entries
    cent, counts = oracle.centroids(entries_np, gid_np, w.g)
    for i, (q, out) in enumerate(zip(batches, outs)):
        problems = compare_lookup(out, entries_np, gid_np, w.g, to_numpy(q), w.k_groups, w.k_entries, 1.0, 0.0,
                                  "bf16", centroid=cent, counts=counts)
        assert not problems, f"batch {i}:\n" + "\n".join(problems[:20])

    from parity import compare_flat

    rows = np.linspace(0, w.b - 1, 8).astype(int)
    problems = compare_flat(flat, entries_np, to_numpy(batches[0]), w.k_entries, 1.0, 0.0, "bf16", rows=rows)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


# ------------------------------------------------------------------ edge cases

@pytest.mark.parametrize("b", [1, 31, 33, 100])
def test_ragged_batches(htam, b):
    entries, gid, centres = _rand_memory(5000, 64, 40, torch.bfloat16, seed=b)
    q = _rand_queries(b, 64, torch.bfloat16, seed=b, centres=centres)
    mem = htam.Memory(entries, gid, 40)
    _check(htam, mem, entries, gid, 40, q, 5, 7)


def test_empty_batch(htam):
    entries, gid, _ = _rand_memory(300, 32, 4, torch.float32, seed=1)
    mem = htam.Memory(entries, gid, 4)
    out = mem.query(torch.empty(0, 32, device=DEV), 2, 3)
    torch.cuda.synchronize()
    assert out["entry_idx"].shape == (0, 3)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_all_groups_selected_is_flat_scan(htam, dtype):
    entries, gid, centres = _rand_memory(3000, 48, 16, dtype, seed=3)
    q = _rand_queries(20, 48, dtype, seed=3, centres=centres)
    mem = htam.Memory(entries, gid, 16)
    out = _check(htam, mem, entries, gid, 16, q, 16, 64)
    assert (out["entry_idx"] >= 0).all()


def test_k_max_both_levels(htam):
    entries, gid, centres = _rand_memory(20000, 128, 100, torch.bfloat16, seed=4)
    q = _rand_queries(64, 128, torch.bfloat16, seed=4, centres=centres)
    mem = htam.Memory(entries, gid, 100)
    _check(htam, mem, entries, gid, 100, q, 64, 64, tau=0.2, eps=0.05)


def test_empty_groups_and_short_candidate_sets(htam):
    # 50 groups declared, only 6 hold entries; k_groups above the non-empty
    # count and k_entries above the candidate-set size both pad.
    gid = torch.tensor([3, 7, 11, 19, 23, 42] * 5, dtype=torch.int32, device=DEV)
    entries, gid, _ = _rand_memory(30, 16, 50, torch.float32, seed=5, clustered=False, gid=gid)
    q = _rand_queries(9, 16, torch.float32, seed=5)
    mem = htam.Memory(entries, gid, 50)
    out = _check(htam, mem, entries, gid, 50, q, 8, 40)
    assert (out["group_idx"][:, 6:] == -1).all()
    assert (out["entry_idx"][:, 30:] == -1).all()


def test_duplicate_rows_tie_to_lower_id(htam):
    base, _, _ = _rand_memory(10, 32, 1, torch.float32, seed=6, clustered=False)
    entries = base.repeat(30, 1).contiguous()  # every row appears 30 times
    gid = (torch.arange(300, device=DEV) % 3).to(torch.int32)
    q = _rand_queries(4, 32, torch.float32, seed=6)
    mem = htam.Memory(entries, gid, 3)
    out = mem.query(q, 3, 20)
    torch.cuda.synchronize()
    ids = out["entry_idx"].cpu().numpy()
    sc = out["entry_score"].cpu().numpy()
    for b in range(4):
        for i in range(19):
            if sc[b, i] == sc[b, i + 1]:
                assert ids[b, i] < ids[b, i + 1]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("min_bucket", [1, 1 << 30])
def test_zero_queries_tie_everything_to_the_lowest_ids(htam, dtype, min_bucket):
    """A zero query scores exactly 0 against every key and entry, in any
    summation order, so both levels are pure ties: the selected groups are
    the lowest non-empty group ids, the entries the lowest entry ids of
    those groups, every candidate weighs 1/n_b and lse = log n_b (any tau).
    Checked exactly on both fine routes (tensor cores / CUDA cores) with
    buckets of several 128-query chunks, and on the flat scan."""
    n, d, g, kg, ke = 5000, 256, 40, 6, 20
    gen = torch.Generator(device=DEV).manual_seed(31)
    pool = torch.tensor([x for x in range(g) if x not in (0, 3, 4)], device=DEV)  # 0, 3, 4 stay empty
    gid = pool[torch.randint(0, pool.numel(), (n,), generator=gen, device=DEV)].to(torch.int32)
    entries, gid, _ = _rand_memory(n, d, g, dtype, seed=31, gid=gid)
    mem = htam.Memory(entries, gid, g)
    mem.set_tensor_core_min_bucket(min_bucket)
    q = torch.zeros(300, d, dtype=dtype, device=DEV)
    out = mem.query(q, kg, ke, tau=0.3, epsilon=0.1)
    flat = mem.query_flat(q, ke, tau=0.3, epsilon=0.1)
    torch.cuda.synchronize()
    gid_np = to_numpy(gid)
    groups = sorted(set(gid_np.tolist()))[:kg]
    cand = np.flatnonzero(np.isin(gid_np, groups))
    assert (out["group_idx"].cpu().numpy() == np.array(groups)).all()
    assert (out["group_score"] == 0).all()
    assert (out["entry_idx"].cpu().numpy() == cand[:ke]).all()
    assert (out["entry_score"] == 0).all()
    torch.testing.assert_close(out["entry_weight"], torch.full_like(out["entry_weight"], 1.0 / cand.size),
                               rtol=1e-5, atol=0)
    torch.testing.assert_close(out["lse"], torch.full_like(out["lse"], float(np.log(cand.size))), rtol=1e-6, atol=0)
    assert (flat["entry_idx"].cpu().numpy() == np.arange(ke)).all()
    torch.testing.assert_close(flat["entry_weight"], torch.full_like(flat["entry_weight"], 1.0 / n), rtol=1e-5, atol=0)
    torch.testing.assert_close(flat["lse"], torch.full_like(flat["lse"], float(np.log(n))), rtol=1e-6, atol=0)
    assert mem.device_status() == htam.HTAM_OK


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("min_bucket", [1, 1 << 30])
def test_large_scores_are_max_shifted(htam, dtype, min_bucket):
    """Rows of norm sqrt(40) and tau = 0.1 give s / tau up to 400, far past
    where exp overflows in fp32 (about 88): the online maximum of the fine
    kernels and the merge's log-sum-exp must keep every weight and lse
    finite and equal to the oracle's.  The tolerance is the bf16 one for
    both dtypes: at this temperature a score's last-place error is
    amplified 10x in the weights."""
    n, d, g, b, kg, ke = 6000, 128, 24, 200, 4, 16
    entries, gid, centres = _rand_memory(n, d, g, torch.float32, seed=41)
    q = _rand_queries(b, d, torch.float32, seed=41, centres=centres)
    scale = float(np.sqrt(40.0))
    entries = (entries * scale).to(dtype).contiguous()
    q = (q * scale).to(dtype).contiguous()
    mem = htam.Memory(entries, gid, g)
    mem.set_tensor_core_min_bucket(min_bucket)
    out = mem.query(q, kg, ke, tau=0.1, epsilon=0.05)
    torch.cuda.synchronize()
    assert mem.device_status() == htam.HTAM_OK
    assert torch.isfinite(out["lse"]).all() and torch.isfinite(out["entry_weight"]).all()
    assert out["lse"].max().item() > 300.0  # the unshifted exponentials would overflow
    problems = compare_lookup(out, to_numpy(entries), to_numpy(gid), g, to_numpy(q), kg, ke, 0.1, 0.05, "bf16")
    assert not problems, "\n".join(problems[:20])


@pytest.mark.parametrize("d", [8, 24, 4096, 16384])
def test_dimension_extremes(htam, d):
    n = 2000 if d <= 4096 else 400
    entries, gid, centres = _rand_memory(n, d, 12, torch.bfloat16, seed=d)
    q = _rand_queries(10, d, torch.bfloat16, seed=d, centres=centres)
    mem = htam.Memory(entries, gid, 12)
    _check(htam, mem, entries, gid, 12, q, 3, 9)


def test_most_groups_and_largest_k(htam):
    """65,536 groups (the most a memory takes), most of them empty or with a
    few entries, k_groups = k_entries = 64; the flat scan and the policy draws
    over all of them."""
    from parity import compare_flat, compare_sampled

    n, g, d = 150000, 65536, 64
    gid = (torch.arange(n, device=DEV, dtype=torch.int64) * 7919 % 50000).to(torch.int32)  # 50,000 non-empty
    entries, gid, centres = _rand_memory(n, d, g, torch.bfloat16, seed=41, gid=gid)
    q = _rand_queries(96, d, torch.bfloat16, seed=41)
    mem = htam.Memory(entries, gid, g)
    rows = np.arange(0, 96, 6)
    _check(htam, mem, entries, gid, g, q, 64, 64, tau=0.3, eps=0.01, rows=rows)
    flat = mem.query_flat(q, 64, tau=0.3, epsilon=0.01)
    torch.cuda.synchronize()
    problems = compare_flat(flat, to_numpy(entries), to_numpy(q), 64, 0.3, 0.01, "bf16", rows=rows)
    assert not problems, "\n".join(problems[:20])
    smp = mem.query_sampled(q, 64, 32, seed=3, offset=4, tau=0.3, epsilon=0.01)
    torch.cuda.synchronize()
    problems = compare_sampled(smp, to_numpy(entries), to_numpy(gid), g, to_numpy(q), 64, 32, 0.3, 0.01, "bf16",
                               seed=3, offset=4, rows=rows)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


def test_large_batch_one_warp_per_query(htam):
    """20,000 queries: selection and merge take one warp per query, and the
    tensor-core buckets hold thousands of queries (many 128-query chunks)."""
    entries, gid, centres = _rand_memory(60000, 128, 400, torch.bfloat16, seed=42)
    q = _rand_queries(20000, 128, torch.bfloat16, seed=42, centres=centres)
    mem = htam.Memory(entries, gid, 400)
    _check(htam, mem, entries, gid, 400, q, 8, 24, tau=0.5, eps=0.02, rows=np.linspace(0, 19999, 40).astype(int))


def test_large_groups_many_segments_ragged_tail(htam):
    # one group of 5,000 rows (40 pages, ragged last page) and a few small ones
    gid = torch.cat([torch.zeros(5000, dtype=torch.int32), torch.arange(1, 6, dtype=torch.int32).repeat(7)])
    gid = gid[torch.randperm(gid.numel(), generator=torch.Generator().manual_seed(0))].to(DEV)
    entries, gid, centres = _rand_memory(gid.numel(), 96, 6, torch.bfloat16, seed=8, gid=gid)
    q = _rand_queries(40, 96, torch.bfloat16, seed=8, centres=centres)
    mem = htam.Memory(entries, gid, 6)
    _check(htam, mem, entries, gid, 6, q, 2, 33)


# ------------------------------------------- tensor-core and CUDA-core paths

TC_CASES = [
    # n, groups, d, batch, k_groups, k_entries: several 128-query chunks per
    # bucket, groups spanning several 16-page segments, ragged last pages
    (60000, 8, 256, 300, 3, 20),
    # d not a multiple of the 64-column K slice; k_entries at the tensor-core limit
    (20000, 50, 1000, 130, 10, 32),
    # one group, one page: a single tile of one page
    (100, 1, 64, 40, 1, 5),
]


@pytest.mark.parametrize("case", TC_CASES)
@pytest.mark.parametrize("min_bucket", [1, 16, 1 << 30])
def test_tensor_core_and_cuda_core_paths(htam, case, min_bucket):
    n, g, d, b, kg, ke = case
    entries, gid, centres = _rand_memory(n, d, g, torch.bfloat16, seed=n + d)
    q = _rand_queries(b, d, torch.bfloat16, seed=n + d, centres=centres)
    mem = htam.Memory(entries, gid, g)
    mem.set_tensor_core_min_bucket(min_bucket)
    mem.read_phase_timing()
    _check(htam, mem, entries, gid, g, q, kg, ke, tau=0.5, eps=0.05)
    ran = mem.read_phase_timing()
    if min_bucket == 1:
        assert ran["fine_tc"][1] > 0
    if min_bucket == 1 << 30:
        assert ran["fine_tc"][1] == 0


@pytest.mark.parametrize("case", TC_CASES[:2])
def test_tensor_core_sm_pairs(htam, case):
    """Buckets of more than 128 queries on SM pairs (cta_group::2: two
    128-query chunks per M=256 MMA, each SM staging half of every entry tile),
    against the oracle and bit for bit against the single-SM kernel."""
    n, g, d, b, kg, ke = case
    entries, gid, centres = _rand_memory(n, d, g, torch.bfloat16, seed=n + d)
    q = _rand_queries(b, d, torch.bfloat16, seed=n + d, centres=centres)
    mem = htam.Memory(entries, gid, g)
    mem.set_tensor_core_min_bucket(1)
    single = mem.query(q, kg, ke, tau=0.5, epsilon=0.05)
    mem.set_tensor_core_pairs(True)
    mem.read_phase_timing()
    out = _check(htam, mem, entries, gid, g, q, kg, ke, tau=0.5, eps=0.05)
    assert mem.read_phase_timing()["fine_tc"][1] == 2  # the pair kernel, then the one-chunk kernel
    for k in ("group_idx", "entry_idx", "entry_score", "entry_weight", "lse"):
        assert torch.equal(out[k], single[k]), k


@pytest.mark.parametrize("b,g,kg", [(512, 64, 8), (513, 64, 8), (64, 2048, 4), (33, 4096, 8)])
def test_bucketing_in_one_block_and_in_five_kernels(htam, b, g, kg):
    """Batches on both sides of the one-block bucketing limits (4,096 rows,
    4,096 bitmap words) against the oracle."""
    entries, gid, centres = _rand_memory(20000, 64, g, torch.bfloat16, seed=b + g)
    q = _rand_queries(b, 64, torch.bfloat16, seed=b + g, centres=centres)
    mem = htam.Memory(entries, gid, g)
    _check(htam, mem, entries, gid, g, q, kg, 12, tau=0.6, eps=0.02, rows=np.linspace(0, b - 1, 24).astype(int))


def test_flat_scan_on_sm_pairs(htam):
    """The flat scan with the SM-pair kernel: every group's bucket holds all
    300 queries (three chunks, the pair of the third one half empty)."""
    from parity import compare_flat

    entries, gid, centres = _rand_memory(30000, 256, 20, torch.bfloat16, seed=51)
    q = _rand_queries(300, 256, torch.bfloat16, seed=51, centres=centres)
    mem = htam.Memory(entries, gid, 20)
    single = mem.query_flat(q, 16, tau=0.5)
    mem.set_tensor_core_pairs(True)
    out = mem.query_flat(q, 16, tau=0.5)
    torch.cuda.synchronize()
    problems = compare_flat(out, to_numpy(entries), to_numpy(q), 16, 0.5, 0.0, "bf16", rows=np.arange(0, 300, 7))
    assert not problems, "\n".join(problems[:20])
    for k in single:
        assert torch.equal(out[k], single[k]), k


def test_append_phase_is_timed_and_counted(htam):
    entries, gid, _ = _rand_memory(2000, 64, 10, torch.bfloat16, seed=52)
    mem = htam.Memory(entries, gid, 10, capacity=3000)
    mem.read_phase_timing()
    mem.set_phase_timing(True)
    e, g, _ = _rand_memory(500, 64, 10, torch.bfloat16, seed=53)
    mem.append(e, g)
    ran = mem.read_phase_timing()
    mem.set_phase_timing(False)
    assert ran["append"][0] > 0 and ran["append"][1] >= 7
    assert ran["queries"] == 0


STREAM_CASES = [
    # n, groups, d, dtype, batch, k_groups, k_entries
    (6000, 30, 4096, torch.bfloat16, 20, 3, 16),   # 8 KiB rows: three ring slots per warp
    (60000, 300, 512, torch.bfloat16, 200, 4, 16), # more work units than SMs: next unit's rows fetched early
    (9000, 40, 1024, torch.bfloat16, 70, 5, 33),   # 2 KiB rows, k_entries above the tensor-core limit
    (5000, 20, 256, torch.float32, 25, 4, 10),     # fp32 rows
    (3000, 12, 2048, torch.float32, 9, 2, 8),      # fp32 8 KiB rows
    (2000, 10, 8192, torch.bfloat16, 6, 2, 5),     # 16 KiB rows: direct loads either way
    (700, 7, 24, torch.bfloat16, 30, 3, 9),        # tiny rows, many per stage
]


@pytest.mark.parametrize("case", STREAM_CASES)
@pytest.mark.parametrize("stream", [0, 1])
def test_cuda_core_rows_streamed_and_loaded_directly(htam, case, stream):
    n, g, d, dtype, b, kg, ke = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + d)
    q = _rand_queries(b, d, dtype, seed=n + d, centres=centres)
    mem = htam.Memory(entries, gid, g)
    mem.set_tensor_core_min_bucket(1 << 30)
    mem.set_stream_rows(stream)
    _check(htam, mem, entries, gid, g, q, kg, ke, tau=0.4, eps=0.02)


PREFIX_CASES = [
    # n, groups, d, dtype, batch, prefix length, lambda, k_groups, k_entries
    (8000, 40, 256, torch.float32, 30, 4, 0.5, 5, 12),
    (20000, 100, 1024, torch.bfloat16, 70, 6, 0.5, 6, 24),
    (6000, 30, 512, torch.bfloat16, 300, 3, 1.3, 4, 16),   # buckets large enough for the tensor cores
    (3000, 12, 512, torch.bfloat16, 9, 1, 0.0, 3, 8),      # one element: the plain lookup
]


@pytest.mark.parametrize("case", PREFIX_CASES)
def test_prefix_query_matches_oracle(htam, case):
    """htam_query_prefix against the oracle's reduced query (Eq. 9 summed over
    the prefix with the Eq. 10 weights), rounded to the memory's dtype the way
    the lookup consumes it, then the oracle lookup."""
    import oracle

    n, g, d, dtype, b, P, lam, kg, ke = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + P)
    prefix = _rand_queries(b * P, d, dtype, seed=n + P, centres=centres).view(b, P, d).contiguous()
    mem = htam.Memory(entries, gid, g)
    out = mem.query_prefix(prefix, lam, kg, ke, tau=0.7, epsilon=0.05)
    torch.cuda.synchronize()
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    qbar = oracle.round_query(oracle.prefix_reduce(to_numpy(prefix), lam), dt)
    problems = compare_lookup(out, to_numpy(entries), to_numpy(gid), g, qbar, kg, ke, 0.7, 0.05, dt)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


def test_prefix_of_one_equals_plain_query_bitwise(htam):
    entries, gid, centres = _rand_memory(5000, 512, 20, torch.bfloat16, seed=3)
    q = _rand_queries(40, 512, torch.bfloat16, seed=3, centres=centres)
    mem = htam.Memory(entries, gid, 20)
    a = mem.query(q, 4, 16, tau=0.5, epsilon=0.1)
    p = mem.query_prefix(q.view(40, 1, 512).contiguous(), 2.0, 4, 16, tau=0.5, epsilon=0.1)
    torch.cuda.synchronize()
    for k in a:
        assert torch.equal(a[k], p[k]), k


def test_prefix_arguments_checked(htam):
    entries, gid, _ = _rand_memory(500, 64, 4, torch.float32, seed=4)
    mem = htam.Memory(entries, gid, 4)
    ok = torch.zeros(3, 2, 64, device=DEV)
    for bad_len in (0, htam.HTAM_MAX_PREFIX + 1):
        pre = torch.zeros(3, max(bad_len, 1), 64, device=DEV)
        if bad_len == 0:
            pre = pre[:, :0, :].contiguous()
        with pytest.raises((htam.HtamError, ValueError)):
            mem.query_prefix(pre, 0.5, 2, 4)
    for lam in (-0.1, float("inf"), float("nan")):
        with pytest.raises(htam.HtamError):
            mem.query_prefix(ok, lam, 2, 4)


EDGE_CASES = [
    # n, groups, d, dtype, batch, prefix length, lambda, features, k_groups, k_entries
    # (batch x prefix > groups forms the whole utility table first)
    (12000, 60, 256, torch.float32, 40, 4, 0.5, 12, 6, 16),
    (20000, 100, 1024, torch.bfloat16, 300, 6, 0.5, 12, 8, 24),   # buckets large enough for the tensor cores
    (5000, 30, 512, torch.bfloat16, 25, 3, 0.0, 5, 4, 8),          # features not a multiple of 4
    (12000, 200, 256, torch.float32, 20, 3, 0.5, 12, 6, 16),       # fewer prefix rows than groups: direct scores
    (12000, 200, 256, torch.float32, 20, 3, 0.5, 7, 6, 16),        # the same with 7 features
]


@pytest.mark.parametrize("case", EDGE_CASES)
def test_edge_routed_lookup_matches_oracle(htam, case):
    """htam_query_edges against the oracle: stage 1 from the edge table (Eq. 9
    with the App. B.6 utility and the Eq. 10 weights), stage 2 from the
    queries on the groups it selected."""
    from parity import compare_edge_lookup

    n, g, d, dtype, b, P, lam, F, kg, ke = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + F)
    q = _rand_queries(b, d, dtype, seed=n + F, centres=centres)
    rng = np.random.default_rng(n + F)
    Z = rng.standard_normal((g, g, F)).astype(np.float32)
    w = rng.standard_normal(F).astype(np.float32)
    prefix = rng.integers(-1, g, (b, P)).astype(np.int32)
    mem = htam.Memory(entries, gid, g)
    out = mem.query_edges(torch.from_numpy(Z).to(DEV), w, prefix, lam, q, kg, ke, tau=0.7, epsilon=0.05)
    torch.cuda.synchronize()
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    problems = compare_edge_lookup(out, to_numpy(entries), to_numpy(gid), g, Z, w.astype(np.float64), prefix, lam,
                                   to_numpy(q), kg, ke, 0.7, 0.05, dt)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


def test_edge_arguments_checked(htam):
    entries, gid, _ = _rand_memory(500, 64, 4, torch.float32, seed=6)
    mem = htam.Memory(entries, gid, 4)
    q = torch.zeros(2, 64, device=DEV)
    Z = torch.zeros(4, 4, 12, device=DEV)
    w = np.ones(12, np.float32)
    good = np.array([[0, -1], [3, 2]], np.int32)
    mem.query_edges(Z, w, good, 0.5, q, 2, 4)
    for bad in (np.array([[0, 4], [1, 2]], np.int32), np.array([[0, -2], [1, 2]], np.int32)):
        with pytest.raises(htam.HtamError):
            mem.query_edges(Z, w, bad, 0.5, q, 2, 4)
    with pytest.raises(htam.HtamError):
        mem.query_edges(torch.zeros(4, 4, htam.HTAM_MAX_EDGE_FEATURES + 1, device=DEV),
                        np.ones(htam.HTAM_MAX_EDGE_FEATURES + 1, np.float32), good, 0.5, q, 2, 4)
    with pytest.raises(htam.HtamError):
        mem.query_edges(Z, np.array([1.0] * 11 + [np.nan], np.float32), good, 0.5, q, 2, 4)


FLAT_CASES = [
    # n, groups, d, dtype, batch, k_entries, tensor-core threshold (None = default)
    (8000, 40, 256, torch.float32, 30, 16, None),        # fp32: CUDA-core kernel
    (20000, 60, 512, torch.bfloat16, 150, 32, None),     # two 128-query chunks per group, the second ragged
    (20000, 60, 512, torch.bfloat16, 150, 33, None),     # k_entries above the tensor-core limit
    (6000, 30, 1024, torch.bfloat16, 7, 12, 1 << 30),    # bf16 rows through the CUDA-core ring
    (30000, 30, 4096, torch.bfloat16, 64, 16, None),     # 8 KiB rows, 64 queries (the 4M workload's batch)
    (60000, 8, 256, torch.bfloat16, 300, 20, None),      # groups spanning many page segments
]


@pytest.mark.parametrize("case", FLAT_CASES)
def test_flat_scan_matches_oracle(htam, case):
    """htam_query_flat against the oracle's flat retrieval (every entry a
    candidate, |C| = n in the epsilon term)."""
    from parity import compare_flat

    n, g, d, dtype, b, ke, tc_min = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + d + b)
    q = _rand_queries(b, d, dtype, seed=n + d + b, centres=centres)
    mem = htam.Memory(entries, gid, g)
    if tc_min is not None:
        mem.set_tensor_core_min_bucket(tc_min)
    mem.read_phase_timing()
    out = mem.query_flat(q, ke, tau=0.6, epsilon=0.05)
    torch.cuda.synchronize()
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    problems = compare_flat(out, to_numpy(entries), to_numpy(q), ke, 0.6, 0.05, dt)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK
    ran = mem.read_phase_timing()
    assert ran["coarse"][1] == 0  # no group stage
    if dtype == torch.bfloat16 and ke <= 32 and tc_min is None:
        assert ran["fine_tc"][1] > 0


@pytest.mark.parametrize("dtype,tc_min", [(torch.bfloat16, None), (torch.bfloat16, 1 << 30), (torch.float32, None)])
def test_flat_scan_equals_lookup_with_every_group(htam, dtype, tc_min):
    """With k_groups = the number of non-empty groups the two-level lookup
    scores the same candidates with the same kernels: identical ids and
    scores.  The softmax denominators are summed over the groups in selection
    order there and in group-id order here, so weights and lse agree to fp32
    rounding."""
    gid = torch.arange(5000, device=DEV, dtype=torch.int32) % 23 * 2  # 23 of 46 groups hold entries
    entries, gid, centres = _rand_memory(5000, 512, 46, dtype, seed=8, gid=gid)
    q = _rand_queries(140, 512, dtype, seed=8)
    mem = htam.Memory(entries, gid, 46)
    if tc_min is not None:
        mem.set_tensor_core_min_bucket(tc_min)
    a = mem.query(q, 23, 24, tau=0.5, epsilon=0.1)
    f = mem.query_flat(q, 24, tau=0.5, epsilon=0.1)
    torch.cuda.synchronize()
    assert torch.equal(a["entry_idx"], f["entry_idx"])
    assert torch.equal(a["entry_score"], f["entry_score"])
    torch.testing.assert_close(f["entry_weight"], a["entry_weight"], rtol=1e-5, atol=1e-9)
    torch.testing.assert_close(f["lse"], a["lse"], rtol=1e-6, atol=1e-6)


def test_flat_scan_short_memory_and_empty_batch(htam):
    """Fewer entries than k_entries pads with -1 / -inf / 0; an empty batch
    launches nothing."""
    gid = torch.tensor([2, 5, 5, 9, 2, 2], dtype=torch.int32, device=DEV)
    entries, gid, _ = _rand_memory(6, 32, 12, torch.float32, seed=9, clustered=False, gid=gid)
    q = _rand_queries(5, 32, torch.float32, seed=9)
    mem = htam.Memory(entries, gid, 12)
    out = mem.query_flat(q, 10, tau=0.3, epsilon=0.2)
    torch.cuda.synchronize()
    from parity import compare_flat

    problems = compare_flat(out, to_numpy(entries), to_numpy(q), 10, 0.3, 0.2, "f32")
    assert not problems, "\n".join(problems)
    assert (out["entry_idx"][:, 6:] == -1).all() and (out["entry_weight"][:, 6:] == 0).all()
    assert torch.isneginf(out["entry_score"][:, 6:]).all()
    empty = mem.query_flat(torch.empty(0, 32, device=DEV), 4)
    torch.cuda.synchronize()
    assert empty["entry_idx"].shape == (0, 4)


def test_flat_scan_after_appends(htam):
    """Appended entries (Eq. 15) are candidates of the next flat scan, also in
    groups that were empty before."""
    from parity import compare_flat

    entries, gid, centres = _rand_memory(3000, 256, 20, torch.bfloat16, seed=10,
                                         gid=torch.arange(3000, device=DEV, dtype=torch.int32) % 10)
    mem = htam.Memory(entries, gid, 20, capacity=6000)
    more, more_gid, _ = _rand_memory(1500, 256, 20, torch.bfloat16, seed=11)
    mem.append(more, more_gid)
    q = _rand_queries(40, 256, torch.bfloat16, seed=10, centres=centres)
    out = mem.query_flat(q, 16, tau=0.8)
    torch.cuda.synchronize()
    all_e = torch.cat([entries, more])
    problems = compare_flat(out, to_numpy(all_e), to_numpy(q), 16, 0.8, 0.0, "bf16")
    assert not problems, "\n".join(problems[:20])


def test_flat_arguments_checked(htam):
    entries, gid, _ = _rand_memory(500, 64, 4, torch.float32, seed=12)
    mem = htam.Memory(entries, gid, 4)
    q = torch.zeros(3, 64, device=DEV)
    for ke in (0, 65):
        with pytest.raises(htam.HtamError):
            mem.query_flat(q, ke)
    for tau, eps in ((0.0, 0.0), (float("nan"), 0.0), (1.0, -0.1), (1.0, 1.5)):
        with pytest.raises(htam.HtamError):
            mem.query_flat(q, 4, tau=tau, epsilon=eps)
    raw = torch.zeros(3 * 64 + 1, device=DEV)
    with pytest.raises(htam.HtamError):  # queries not 16-byte aligned
        mem.query_flat(raw[1:].view(3, 64), 4)


SAMPLED_CASES = [
    # n, groups, d, dtype, batch, k_groups, k_entries, tau, eps
    (8000, 40, 256, torch.float32, 30, 5, 12, 0.3, 0.1),
    (20000, 100, 512, torch.bfloat16, 300, 1, 16, 0.05, 0.0),   # the paper's single draw; tensor-core buckets
    (20000, 100, 512, torch.bfloat16, 70, 8, 24, 0.5, 0.3),
    (6000, 50, 128, torch.bfloat16, 40, 6, 8, 1.0, 1.0),        # pure exploration: uniform over G_t
    (3000, 1000, 64, torch.float32, 9, 64, 16, 0.2, 0.05),      # many groups, most of them empty or small
]


@pytest.mark.parametrize("case", SAMPLED_CASES)
def test_sampled_lookup_matches_oracle(htam, case):
    """htam_query_sampled against the oracle: the draws are the top k_groups
    of the oracle's policy keys (Eq. 11 with the same Philox uniforms), the
    group scores q . c_g, and stage 2 over the drawn groups."""
    from parity import compare_sampled

    n, g, d, dtype, b, kg, ke, tau, eps = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + b)
    q = _rand_queries(b, d, dtype, seed=n + b, centres=centres)
    mem = htam.Memory(entries, gid, g)
    out = mem.query_sampled(q, kg, ke, seed=1234 + n, offset=5, tau=tau, epsilon=eps)
    torch.cuda.synchronize()
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    problems = compare_sampled(out, to_numpy(entries), to_numpy(gid), g, to_numpy(q), kg, ke, tau, eps, dt,
                               seed=1234 + n, offset=5)
    assert not problems, "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


def test_sampled_draws_follow_the_policy(htam):
    """One query repeated 20,000 times: each copy draws with its own uniforms,
    so the first draws are distributed as mu_g of Eq. 11 (chi-square against
    the oracle's policy over the GPU's own group keys), and the empty group
    never comes up."""
    import oracle
    from scipy import stats

    gid = torch.tensor([0, 1, 2, 3, 5, 6] * 50, dtype=torch.int32, device=DEV)  # group 4 empty
    entries, gid, _ = _rand_memory(300, 32, 7, torch.float32, seed=13, gid=gid)
    q = _rand_queries(1, 32, torch.float32, seed=13).repeat(20000, 1).contiguous()
    mem = htam.Memory(entries, gid, 7)
    out = mem.query_sampled(q, 1, 4, seed=77, offset=0, tau=0.1, epsilon=0.2)
    torch.cuda.synchronize()
    first = out["group_idx"][:, 0].cpu().numpy()
    keys_f32 = mem.group_keys().double().numpy()
    s = oracle.coarse_scores(to_numpy(q[:1]), keys_f32)
    counts = mem.group_counts().numpy()
    _, mu = oracle.policy_keys(s, counts, 0.1, 0.2, 0, 0)
    obs = np.bincount(first, minlength=7)
    assert obs[4] == 0
    ne = counts > 0
    assert stats.chisquare(obs[ne], 20000 * mu[0][ne] / mu[0][ne].sum()).pvalue > 1e-4


def test_sampled_draws_are_reproducible_and_offset_dependent(htam):
    entries, gid, centres = _rand_memory(6000, 256, 40, torch.bfloat16, seed=14)
    q = _rand_queries(64, 256, torch.bfloat16, seed=14, centres=centres)
    mem = htam.Memory(entries, gid, 40)
    a = mem.query_sampled(q, 4, 16, seed=5, offset=100, tau=0.5, epsilon=0.1)
    b = mem.query_sampled(q, 4, 16, seed=5, offset=100, tau=0.5, epsilon=0.1)
    c = mem.query_sampled(q, 4, 16, seed=5, offset=101, tau=0.5, epsilon=0.1)
    d = mem.query_sampled(q, 4, 16, seed=6, offset=100, tau=0.5, epsilon=0.1)
    torch.cuda.synchronize()
    for k in a:
        assert torch.equal(a[k], b[k]), k
    assert not torch.equal(a["group_idx"], c["group_idx"])
    assert not torch.equal(a["group_idx"], d["group_idx"])


def test_cold_policy_draws_what_the_ranking_selects(htam):
    """tau -> 0 with no exploration: the draws are stage 1's ranking."""
    entries, gid, centres = _rand_memory(8000, 128, 60, torch.float32, seed=15)
    q = _rand_queries(50, 128, torch.float32, seed=15, centres=centres)
    mem = htam.Memory(entries, gid, 60)
    a = mem.query(q, 6, 10, tau=1e-4)
    s = mem.query_sampled(q, 5, 10, seed=1, offset=2, tau=1e-4)
    torch.cuda.synchronize()
    # Rows whose six best groups are 2e-3 apart (20 units of key next to the
    # Gumbel noise, which exceeds that with probability about e^-20).
    gaps = (a["group_score"][:, :-1] - a["group_score"][:, 1:]).min(dim=1).values
    clear = gaps > 2e-3
    assert clear.sum() > 10
    assert torch.equal(a["group_idx"][clear][:, :5], s["group_idx"][clear])


def test_sampled_edge_routed_lookup_matches_oracle(htam):
    """htam_query_edges_sampled: the draws from the policy over the edge-table
    scores (Eq. 9 with the App. B.6 utility), stage 2 over them."""
    import oracle
    from parity import compare_sampled

    n, g, d, b, P, F, kg, ke = 12000, 60, 256, 40, 4, 12, 3, 16
    entries, gid, centres = _rand_memory(n, d, g, torch.float32, seed=16)
    q = _rand_queries(b, d, torch.float32, seed=16, centres=centres)
    rng = np.random.default_rng(16)
    Z = rng.standard_normal((g, g, F)).astype(np.float32)
    w = rng.standard_normal(F).astype(np.float32)
    prefix = rng.integers(-1, g, (b, P)).astype(np.int32)
    mem = htam.Memory(entries, gid, g)
    out = mem.query_edges(torch.from_numpy(Z).to(DEV), w, prefix, 0.5, q, kg, ke, tau=0.7, epsilon=0.1,
                          sampling=(42, 9))
    torch.cuda.synchronize()
    scores = oracle.edge_scores(Z, w.astype(np.float64), prefix, 0.5)
    mag = oracle.edge_scores(np.abs(Z), np.abs(w.astype(np.float64)), prefix, 0.5)
    problems = compare_sampled(out, to_numpy(entries), to_numpy(gid), g, to_numpy(q), kg, ke, 0.7, 0.1, "f32",
                               seed=42, offset=9, scores=scores, score_tol=edge_score_tol(scores, mag, F, P))
    assert not problems, "\n".join(problems[:20])


def test_sampled_zipf_1m_workload_sampled_rows(htam):
    """Full size, full batch (4,096 queries against 1,048,576 entries in
    1,024 groups), a sample of the queries checked."""
    from parity import compare_sampled

    w = workloads.WORKLOADS["zipf_bf16_1m"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    q = workloads.make_queries(w, gid, centres, seed=0)
    mem = htam.Memory(entries, gid, w.g)
    out = mem.query_sampled(q, w.k_groups, w.k_entries, seed=2026, offset=3, tau=0.5, epsilon=0.05)
    torch.cuda.synchronize()
    rows = np.linspace(0, w.b - 1, 24).astype(int)
    problems = compare_sampled(out, to_numpy(entries), to_numpy(gid), w.g, to_numpy(q), w.k_groups, w.k_entries,
                               0.5, 0.05, "bf16", seed=2026, offset=3, rows=rows)
    assert not problems, "\n".join(problems[:20])


def test_tuning_defaults_follow_row_length_and_round_trip(htam):
    """The tensor-core threshold defaults to 2 queries for every row length;
    values set are read back; bad keys and values are refused."""
    for d, want in ((1024, 2), (2048, 2), (4096, 2)):
        e, gid, _ = _rand_memory(300, d, 3, torch.bfloat16, seed=d)
        mem = htam.Memory(e, gid, 3)
        assert mem.get_tuning(htam.HTAM_TUNE_TC_MIN_BUCKET) == want
        assert mem.get_tuning(htam.HTAM_TUNE_STREAM_ROWS) == 1
        assert mem.get_tuning(htam.HTAM_TUNE_TC_PAIRS) == 0
        mem.set_tensor_core_min_bucket(7)
        mem.set_stream_rows(False)
        mem.set_tensor_core_pairs(True)
        assert mem.get_tuning(htam.HTAM_TUNE_TC_MIN_BUCKET) == 7
        assert mem.get_tuning(htam.HTAM_TUNE_STREAM_ROWS) == 0
        assert mem.get_tuning(htam.HTAM_TUNE_TC_PAIRS) == 1
        with pytest.raises(htam.HtamError):
            mem.set_tuning(htam.HTAM_TUNE_TC_PAIRS, 2)
        with pytest.raises(htam.HtamError):
            mem.get_tuning(99)
        with pytest.raises(htam.HtamError):
            mem.set_tuning(htam.HTAM_TUNE_TC_MIN_BUCKET, 0)


@pytest.mark.parametrize("min_bucket", [2, 1 << 30])
def test_two_query_buckets_on_both_paths(htam, min_bucket):
    """Buckets of two or three queries (the smallest the tensor cores take by
    default) scored on the tensor cores and on the CUDA cores."""
    entries, gid, centres = _rand_memory(20000, 1024, 400, torch.bfloat16, seed=41)
    q = _rand_queries(60, 1024, torch.bfloat16, seed=41, centres=centres)
    mem = htam.Memory(entries, gid, 400)
    mem.set_tensor_core_min_bucket(min_bucket)
    _check(htam, mem, entries, gid, 400, q, 6, 24, tau=0.5, eps=0.1)


@pytest.mark.parametrize("min_bucket", [1, 1 << 30])
def test_duplicate_bf16_rows_tie_to_lower_id_on_both_paths(htam, min_bucket):
    """Exactly equal scores (duplicate rows spread over pages and chunks)
    must come out in entry-id order on both fine kernels."""
    base, _, _ = _rand_memory(40, 128, 1, torch.bfloat16, seed=22, clustered=False)
    entries = base.repeat(100, 1).contiguous()            # 4,000 rows, each value 100 times
    gid = (torch.arange(4000, device=DEV) % 2).to(torch.int32)
    q = _rand_queries(50, 128, torch.bfloat16, seed=22)
    mem = htam.Memory(entries, gid, 2)
    mem.set_tensor_core_min_bucket(min_bucket)
    _check(htam, mem, entries, gid, 2, q, 2, 32)
    out = mem.query(q, 2, 32)
    torch.cuda.synchronize()
    ids, sc = out["entry_idx"].cpu().numpy(), out["entry_score"].cpu().numpy()
    for b in range(50):
        for i in range(31):
            assert sc[b, i] > sc[b, i + 1] or (sc[b, i] == sc[b, i + 1] and ids[b, i] < ids[b, i + 1])


def test_paths_agree_on_the_zipf_65k_workload(htam):
    w = workloads.WORKLOADS["zipf_bf16_65k"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    q = workloads.make_queries(w, gid, centres, seed=0)
    mem = htam.Memory(entries, gid, w.g)
    outs = []
    for min_bucket in (1, 1 << 30):
        mem.set_tensor_core_min_bucket(min_bucket)
        outs.append({k: v.clone() for k, v in mem.query(q, w.k_groups, w.k_entries).items()})
    torch.cuda.synchronize()
    assert torch.equal(outs[0]["group_idx"], outs[1]["group_idx"])
    same = (outs[0]["entry_idx"] == outs[1]["entry_idx"]).float().mean().item()
    assert same > 0.99
    torch.testing.assert_close(outs[0]["lse"], outs[1]["lse"], rtol=1e-4, atol=1e-4)


# ---------------------------------------------------------------- append path

@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_append_rounds_match_rebuilt_oracle(htam, dtype):
    entries, gid, centres = _rand_memory(4000, 64, 30, dtype, seed=9)
    mem = htam.Memory(entries, gid, 30, capacity=4000 + 3 * 700)
    q = _rand_queries(50, 64, dtype, seed=9, centres=centres)
    all_e, all_g = entries, gid
    for r in range(3):
        new_e, new_g, _ = _rand_memory(700, 64, 30, dtype, seed=100 + r)
        mem.append(new_e, new_g)
        all_e = torch.cat([all_e, new_e])
        all_g = torch.cat([all_g, new_g])
        assert mem.info()["n"] == all_e.shape[0]
        assert (mem.group_counts().numpy() == np.bincount(to_numpy(all_g), minlength=30)).all()
        _check(htam, mem, all_e, all_g, 30, q, 4, 12, tau=0.3)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_memory_built_empty_then_filled_by_appends(htam, dtype):
    """A memory built with no entries has no non-empty group, so a lookup
    returns padding only (lse = -inf: an empty candidate set).  Appends then
    fill half of the groups, and later all of them: groups that were empty
    become selectable, and each lookup matches the oracle on the rows
    appended so far (ids count from 0 in append order).  The appends fill
    the capacity exactly; one more row is refused."""
    d, g = 64, 12
    mem = htam.Memory(torch.empty(0, d, dtype=dtype, device=DEV), torch.empty(0, dtype=torch.int32, device=DEV),
                      g, capacity=2400)  # the two appends below fill it exactly
    gen = torch.Generator(device=DEV).manual_seed(21)
    centres = torch.randn(g, d, generator=gen, device=DEV)
    q = _rand_queries(40, d, dtype, seed=21, centres=centres)
    out = mem.query(q, 3, 5)
    torch.cuda.synchronize()
    assert (out["group_idx"] == -1).all() and torch.isneginf(out["group_score"]).all()
    assert (out["entry_idx"] == -1).all() and (out["entry_weight"] == 0).all()
    assert torch.isneginf(out["entry_score"]).all() and torch.isneginf(out["lse"]).all()
    assert mem.device_status() == htam.HTAM_OK

    half = torch.randint(0, g // 2, (900,), generator=gen, device=DEV, dtype=torch.int64).to(torch.int32)
    rounds = [half, torch.randint(0, g, (1500,), generator=gen, device=DEV, dtype=torch.int64).to(torch.int32)]
    all_e, all_g = [], []
    for r, gid in enumerate(rounds):
        x = centres[gid.long()] + 0.3 * torch.randn(gid.shape[0], d, generator=gen, device=DEV)
        e = _unit(x).to(dtype).contiguous()
        mem.append(e, gid)
        all_e.append(e)
        all_g.append(gid)
        ents, gids = torch.cat(all_e), torch.cat(all_g)
        assert mem.info()["n"] == ents.shape[0]
        counts = np.bincount(to_numpy(gids), minlength=g)
        assert (mem.group_counts().numpy() == counts).all()
        import oracle

        keys = mem.group_keys().double().numpy()
        ref, _ = oracle.centroids(to_numpy(ents), to_numpy(gids), g)
        filled = counts > 0  # the oracle's mean of an empty group is NaN
        np.testing.assert_allclose(keys[filled], ref[filled], rtol=1e-5, atol=1e-6)  # fp32 means
        assert (keys[~filled] == 0).all()  # the library's rows of empty groups are zero
        out = _check(htam, mem, ents, gids, g, q, 4, 8, tau=0.5, eps=0.05)
        selected = out["group_idx"].cpu()
        if r == 0:  # only the filled half can be selected; the rest pads
            assert ((selected >= 0) & (selected < g // 2)).sum(1).eq(4).all()
        else:
            assert (selected >= g // 2).any()
    one = torch.zeros(1, d, dtype=dtype, device=DEV)
    with pytest.raises(htam.HtamError) as err:
        mem.append(one, torch.zeros(1, dtype=torch.int32, device=DEV))
    assert err.value.status == htam.HTAM_ECAPACITY and mem.info()["n"] == 2400


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_appends_queued_back_to_back_grow_one_group(htam, dtype):
    """Appends run on the device with no host round trip, so the host sizes
    a query's scratch from group sizes that may lag behind the queued
    appends.  Eight batches of 3,000 rows all go to group 0 (24,000 rows,
    188 new pages), each followed at once by a lookup that selects it, with
    nothing synchronised in between; every lookup is then checked against
    the oracle over the memory as it stood at that point."""
    d, g = 64, 10
    entries, gid, centres = _rand_memory(2000, d, g, dtype, seed=40)
    mem = htam.Memory(entries, gid, g, capacity=2000 + 8 * 3000)
    gen = torch.Generator(device=DEV).manual_seed(41)
    q = _rand_queries(48, d, dtype, seed=40, centres=centres)
    all_e, all_g, outs = [entries], [gid], []
    for r in range(8):
        new_g = torch.zeros(3000, dtype=torch.int32, device=DEV)
        x = centres[0] + 0.3 * torch.randn(3000, d, generator=gen, device=DEV)
        new_e = _unit(x).to(dtype).contiguous()
        mem.append(new_e, new_g)
        all_e.append(new_e)
        all_g.append(new_g)
        outs.append(({k: v.clone() for k, v in mem.query(q, 3, 12, tau=0.5).items()}, len(all_e)))
    torch.cuda.synchronize()
    assert mem.device_status() == htam.HTAM_OK
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    for r, (out, upto) in enumerate(outs):
        ents, gids = torch.cat(all_e[:upto]), torch.cat(all_g[:upto])
        assert (out["group_idx"] == 0).any()  # the grown group is selected
        problems = compare_lookup(out, to_numpy(ents), to_numpy(gids), g, to_numpy(q), 3, 12, 0.5, 0.0, dt)
        assert not problems, f"lookup after append {r}:\n" + "\n".join(problems[:20])
    assert mem.info()["n"] == 2000 + 8 * 3000


def test_append_updates_group_keys_in_place(htam):
    import oracle

    entries, gid, _ = _rand_memory(3000, 32, 8, torch.float32, seed=10)
    mem = htam.Memory(entries, gid, 8, capacity=6000)
    new_e, new_g, _ = _rand_memory(2500, 32, 8, torch.float32, seed=11)
    mem.append(new_e, new_g)
    keys = mem.group_keys().numpy()
    ref, _ = oracle.centroids(to_numpy(torch.cat([entries, new_e])), to_numpy(torch.cat([gid, new_g])), 8)
    np.testing.assert_allclose(keys, ref, rtol=1e-6, atol=1e-7)


def test_append_errors_leave_memory_unchanged(htam):
    entries, gid, centres = _rand_memory(1000, 32, 10, torch.bfloat16, seed=12)
    mem = htam.Memory(entries, gid, 10, capacity=1100)
    q = _rand_queries(8, 32, torch.bfloat16, seed=12, centres=centres)
    before = {k: v.clone() for k, v in mem.query(q, 3, 5).items()}
    bad_e, bad_g, _ = _rand_memory(50, 32, 10, torch.bfloat16, seed=13)
    bad_g[17] = 10  # out of range: found on the device, reported by the status call
    mem.append(bad_e, bad_g)
    after_bad = {k: v.clone() for k, v in mem.query(q, 3, 5).items()}  # queued behind the rejected batch
    assert mem.device_status() == htam.HTAM_EINVAL
    assert mem.device_status() == htam.HTAM_OK  # read and cleared
    with pytest.raises(htam.HtamError) as err:
        mem.append(bad_e, bad_g, check=True)
    assert err.value.status == htam.HTAM_EINVAL
    big_e, big_g, _ = _rand_memory(101, 32, 10, torch.bfloat16, seed=14)
    with pytest.raises(htam.HtamError) as err:
        mem.append(big_e, big_g)
    assert err.value.status == htam.HTAM_ECAPACITY
    after = mem.query(q, 3, 5)
    torch.cuda.synchronize()
    assert mem.info()["n"] == 1000
    assert (mem.group_counts().numpy() == np.bincount(to_numpy(gid), minlength=10)).all()
    for k in before:
        assert torch.equal(before[k], after[k]) and torch.equal(before[k], after_bad[k])
    # The rejected batches left the id numbering alone: the next rows are 1000..
    ok_e, ok_g, _ = _rand_memory(100, 32, 10, torch.bfloat16, seed=15)
    mem.append(ok_e, ok_g, check=True)
    _check(htam, mem, torch.cat([entries, ok_e]), torch.cat([gid, ok_g]), 10, q, 3, 5)


NEAREST_CASES = [
    # n, groups, d, dtype, appended rows, share without a group
    (4000, 30, 64, torch.float32, 700, 0.5),
    (6000, 40, 512, torch.bfloat16, 1500, 1.0),     # every row assigned, tensor-core scores
    (3000, 2000, 64, torch.bfloat16, 5000, 0.7),    # rows x groups > 4M: three passes, the last ragged
]


@pytest.mark.parametrize("case", NEAREST_CASES)
def test_append_without_group_joins_nearest_key(htam, case):
    """Appended rows with group id -1 join the group whose key (before the
    append) scores highest against them, ranked like stage 1 (the index rule
    on the oracle's float64 scores); given ids are kept; the memory then
    answers like the oracle rebuilt with the assigned ids."""
    import oracle
    from parity import check_ranked

    n, g, d, dtype, add, share = case
    entries, gid, centres = _rand_memory(n, d, g, dtype, seed=n + add)
    mem = htam.Memory(entries, gid, g, capacity=n + add)
    new_e, new_g, _ = _rand_memory(add, d, g, dtype, seed=n + add + 1)
    drop = torch.rand(add, generator=torch.Generator(device=DEV).manual_seed(3), device=DEV) < share
    new_g = torch.where(drop, torch.full_like(new_g, -1), new_g).contiguous()
    cent, counts = oracle.centroids(to_numpy(entries), to_numpy(gid), g)
    assigned = mem.append_assign(new_e, new_g)
    torch.cuda.synchronize()
    a = to_numpy(assigned)
    given = to_numpy(new_g)
    assert (a[given >= 0] == given[given >= 0]).all()
    miss = np.flatnonzero(given == -1)
    ref_gi, ref_gs = oracle.stage1(to_numpy(new_e)[miss], cent, counts, min(2, g))
    xf = to_numpy(new_e)[miss]
    xf = (xf.astype(np.uint32) << 16).view(np.float32).astype(np.float64) if xf.dtype == np.uint16 else xf.astype(np.float64)
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    problems = []
    for r, i in enumerate(miss):
        problems += check_ranked(f"row {i}", [a[i]], [float(cent[a[i]] @ xf[r])], ref_gi[r], ref_gs[r], 1,
                                 lambda gg, r=r: float(cent[gg] @ xf[r]), dt)
    assert not problems, "\n".join(problems[:20])
    all_e = torch.cat([entries, new_e])
    all_g = torch.cat([gid, assigned])
    assert (mem.group_counts().numpy() == np.bincount(to_numpy(all_g), minlength=g)).all()
    q = _rand_queries(40, d, dtype, seed=n, centres=centres)
    _check(htam, mem, all_e, all_g, g, q, min(4, g), 12, tau=0.4)


def test_append_without_group_in_place_and_plain_append(htam):
    """The assigned ids may overwrite the input ids; htam_append_transitions
    takes -1 the same way."""
    entries, gid, _ = _rand_memory(2000, 64, 12, torch.float32, seed=21)
    mem_a = htam.Memory(entries, gid, 12, capacity=3000)
    mem_b = htam.Memory(entries, gid, 12, capacity=3000)
    new_e, _, _ = _rand_memory(500, 64, 12, torch.float32, seed=22)
    ids = torch.full((500,), -1, dtype=torch.int32, device=DEV)
    ids[::3] = 5
    ref = mem_a.append_assign(new_e, ids.clone())
    mem_b.append(new_e, ids)
    import ctypes

    from paper_2605_29734_gb300.htam import _dev_ptr, _lib, _stream_ptr

    mem_c = htam.Memory(entries, gid, 12, capacity=3000)
    inplace = ids.clone()
    assert _lib.htam_append_assign(mem_c.handle, _dev_ptr(new_e), _dev_ptr(inplace), 500, _dev_ptr(inplace),
                                   _stream_ptr(None)) == htam.HTAM_OK
    torch.cuda.synchronize()
    assert torch.equal(inplace, ref)
    assert (mem_a.group_counts() == mem_b.group_counts()).all()
    assert (mem_c.group_counts() == mem_b.group_counts()).all()


def test_append_without_group_errors(htam):
    """-1 into a memory with no entries has no key to join (EINVAL); ids
    below -1 stay invalid; the memory is unchanged."""
    empty = htam.Memory(torch.empty(0, 32, device=DEV), torch.empty(0, dtype=torch.int32, device=DEV), 5,
                        capacity=100)
    e, _, _ = _rand_memory(10, 32, 5, torch.float32, seed=23)
    with pytest.raises(htam.HtamError) as err:
        empty.append(e, torch.full((10,), -1, dtype=torch.int32, device=DEV), check=True)
    assert err.value.status == htam.HTAM_EINVAL
    assert empty.info()["n"] == 0
    entries, gid, _ = _rand_memory(100, 32, 5, torch.float32, seed=24)
    mem = htam.Memory(entries, gid, 5, capacity=200)
    bad = torch.full((10,), -1, dtype=torch.int32, device=DEV)
    bad[4] = -2
    with pytest.raises(htam.HtamError) as err:
        mem.append(e, bad, check=True)
    assert err.value.status == htam.HTAM_EINVAL
    assert mem.info()["n"] == 100
    assert (mem.group_counts().numpy() == np.bincount(to_numpy(gid), minlength=5)).all()


def test_stream_workload_all_rounds(htam):
    """The streaming workload as the benchmark runs it: 100 rounds, each
    appending 4,096 clustered rows (the memory update of Eq. 15, keys updated
    in place) and then answering 1,024 queries (the benchmark's four batches
    in turn), the memory growing from 524,288 to 933,888 entries.  Every 10th
    round all 1,024 queries are checked against the oracle over the memory
    as it stands (group keys accumulated incrementally in float64)."""
    import oracle

    w = workloads.WORKLOADS["stream_bf16_512k"]
    entries, gid, centres = workloads.make_memory(w, seed=0, device=DEV)
    mem = htam.Memory(entries, gid, w.g, capacity=w.capacity)
    batches = _bench_batches(w, gid, centres)
    all_e, all_g = [to_numpy(entries)], [to_numpy(gid)]
    acc = oracle.CentroidAccumulator(w.g, w.d)
    acc.add(all_e[0], all_g[0])
    for r in range(w.rounds):
        new_e, new_g = workloads.make_append_batch(w, centres, r, seed=0, device=DEV)
        mem.append(new_e, new_g)
        all_e.append(to_numpy(new_e))
        all_g.append(to_numpy(new_g))
        acc.add(all_e[-1], all_g[-1])
        q = batches[r % len(batches)]
        out = mem.query(q, w.k_groups, w.k_entries)
        if r % 10 != 9:
            continue
        torch.cuda.synchronize()
        cent, counts = acc.finalize()
        e_np, g_np = np.concatenate(all_e), np.concatenate(all_g)
        assert mem.info()["n"] == e_np.shape[0] == w.n + (r + 1) * w.append_per_round
        assert (mem.group_counts().numpy() == counts).all()
        problems = compare_lookup(out, e_np, g_np, w.g, to_numpy(q), w.k_groups, w.k_entries, 1.0, 0.0,
                                  "bf16", centroid=cent, counts=counts)
        assert not problems, f"round {r}:\n" + "\n".join(problems[:20])
    assert mem.device_status() == htam.HTAM_OK


# ------------------------------------------------------------------ interfaces

def test_host_buffer_query_matches_device_query(htam):
    entries, gid, centres = _rand_memory(8000, 128, 20, torch.bfloat16, seed=15)
    q = _rand_queries(70, 128, torch.bfloat16, seed=15, centres=centres)
    mem = htam.Memory(entries, gid, 20)
    dev = mem.query(q, 4, 10, tau=0.7, epsilon=0.2)
    host = mem.query_host(q.cpu().pin_memory(), 4, 10, tau=0.7, epsilon=0.2)
    for k in dev:
        assert torch.equal(dev[k].cpu(), host[k]), k


def test_repeated_queries_are_bitwise_deterministic(htam):
    entries, gid, centres = _rand_memory(30000, 256, 64, torch.bfloat16, seed=16)
    q = _rand_queries(200, 256, torch.bfloat16, seed=16, centres=centres)
    mem = htam.Memory(entries, gid, 64)
    a = {k: v.clone() for k, v in mem.query(q, 8, 16).items()}
    mem2 = htam.Memory(entries, gid, 64)
    b = mem2.query(q, 8, 16)
    c = mem.query(q, 8, 16)
    torch.cuda.synchronize()
    for k in a:
        assert torch.equal(a[k], b[k]) and torch.equal(a[k], c[k]), k


def test_programmatic_launch_on_and_off_agree_bitwise(htam):
    """Kernels launched with programmatic stream serialisation (the default)
    and plainly give bit-identical lookups and appends: every kernel waits
    for its predecessor before touching memory either way."""
    entries, gid, centres = _rand_memory(30000, 256, 64, torch.bfloat16, seed=26)
    q = _rand_queries(300, 256, torch.bfloat16, seed=26, centres=centres)
    extra, extra_g, _ = _rand_memory(2000, 256, 64, torch.bfloat16, seed=27)
    outs = []
    for pdl in (1, 0):
        mem = htam.Memory(entries, gid, 64, capacity=32000)
        mem.set_programmatic_launch(pdl)
        a = {k: v.clone() for k, v in mem.query(q, 8, 16).items()}
        mem.append(extra, extra_g)
        b = {k: v.clone() for k, v in mem.query(q, 8, 16).items()}
        outs.append((a, b, mem.group_keys()))
        assert mem.device_status() == htam.HTAM_OK
    for x, y in zip(outs[0][:2], outs[1][:2]):
        for k in x:
            assert torch.equal(x[k], y[k]), k
    assert torch.equal(outs[0][2], outs[1][2])


def test_query_rows_copied_or_gathered_agree_bitwise(htam):
    """The tensor-core kernel takes its query rows from the query matrix by
    its copier warp for batches of up to 2,048 queries, and from a
    bucket-ordered copy by TMA above that.  The same 2,048 queries give
    bit-identical results either way: once alone (copier), once followed by
    a repeat of the batch (4,096 queries, TMA), every bucket on the tensor
    cores in both."""
    entries, gid, centres = _rand_memory(40000, 256, 96, torch.bfloat16, seed=61)
    q = _rand_queries(2048, 256, torch.bfloat16, seed=61, centres=centres)
    mem = htam.Memory(entries, gid, 96)
    mem.set_tensor_core_min_bucket(1)
    a = {k: v.clone() for k, v in mem.query(q, 6, 16, tau=0.5, epsilon=0.05).items()}
    b = mem.query(torch.cat([q, q]).contiguous(), 6, 16, tau=0.5, epsilon=0.05)
    torch.cuda.synchronize()
    for k in a:
        assert torch.equal(a[k], b[k][:2048]) and torch.equal(a[k], b[k][2048:]), k
    assert mem.device_status() == htam.HTAM_OK


def test_bad_query_arguments(htam):
    entries, gid, _ = _rand_memory(100, 16, 4, torch.float32, seed=17)
    mem = htam.Memory(entries, gid, 4)
    q = _rand_queries(2, 16, torch.float32, seed=17)
    for kw in (dict(k_groups=0, k_entries=1), dict(k_groups=5, k_entries=1), dict(k_groups=1, k_entries=65),
               dict(k_groups=1, k_entries=1, tau=0.0), dict(k_groups=1, k_entries=1, epsilon=1.5)):
        with pytest.raises(htam.HtamError) as err:
            mem.query(q, **kw)
        assert err.value.status == htam.HTAM_EINVAL


def test_bounded_wait_gives_up_and_context_survives(htam):
    assert htam.selftest_wait_timeout(1000) == htam.HTAM_ETIMEOUT
    entries, gid, _ = _rand_memory(500, 16, 4, torch.float32, seed=18)
    mem = htam.Memory(entries, gid, 4)
    q = _rand_queries(3, 16, torch.float32, seed=18)
    _check(htam, mem, entries, gid, 4, q, 2, 4)


def test_build_rejects_out_of_range_group_ids(htam):
    entries, gid, _ = _rand_memory(100, 16, 4, torch.float32, seed=19)
    gid[5] = -1
    with pytest.raises(htam.HtamError) as err:
        htam.Memory(entries, gid, 4)
    assert err.value.status == htam.HTAM_EINVAL
