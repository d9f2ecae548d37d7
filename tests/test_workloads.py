"""The seeded input recipe (CPU): group sizes, shuffled group ids, unit-norm
rows, queries drawn in proportion to group size, append batches.  These are
the shapes and distributions every parity test and the benchmark use."""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2605_29734_gb300 import workloads
from paper_2605_29734_gb300.workloads import zipf_sizes


@pytest.mark.parametrize("n,g,lo,hi", [(65536, 256, 31, 13483), (1048576, 1024, 93, 187577),
                                       (524288, 512, 106, 100224)])
def test_zipf_sizes(n, g, lo, hi):
    """n_r = 1 + the largest-remainder share of the other n - G entries in
    proportion to r^-1.1: the sum is exact, every group has an entry, sizes
    fall with rank, and each share is its exact value rounded down or up,
    the ups going to the largest remainders."""
    s = zipf_sizes(n, g)
    assert s.sum() == n and s.min() == lo and s.max() == hi
    assert (s[:-1] >= s[1:]).all()
    w = np.arange(1, g + 1, dtype=np.float64) ** -1.1
    share = w / w.sum() * (n - g)
    extra = s - 1 - np.floor(share)
    assert set(np.unique(extra)) <= {0, 1}
    frac = share - np.floor(share)
    if 0 < extra.sum() < g:
        assert frac[extra == 1].min() >= frac[extra == 0].max()


def test_zipf_sizes_need_an_entry_per_group():
    with pytest.raises(ValueError):
        zipf_sizes(10, 11)


def test_group_ids_follow_the_sizes_in_shuffled_order():
    w = dataclasses.replace(workloads.WORKLOADS["zipf_bf16_65k"], n=20000, g=200)
    gid = workloads.make_group_ids(w, seed=0).numpy()
    assert gid.dtype == np.int32 and gid.shape == (20000,)
    assert (np.bincount(gid, minlength=200) == zipf_sizes(20000, 200)).all()
    assert (np.diff(gid) < 0).any()  # not grouped: a build must sort
    again = workloads.make_group_ids(w, seed=0).numpy()
    assert (gid == again).all()
    assert (gid != workloads.make_group_ids(w, seed=1).numpy()).any()


def test_uniform_and_uniform_random_group_ids():
    w = dataclasses.replace(workloads.WORKLOADS["uniform_bf16_4m"], n=4096, g=64, d=64)
    assert (np.bincount(workloads.make_group_ids(w).numpy(), minlength=64) == 64).all()
    t = workloads.WORKLOADS["tiny_f32_1k"]
    gid = workloads.make_group_ids(t).numpy()
    assert gid.min() >= 0 and gid.max() < t.g and len(np.unique(gid)) > t.g // 2


@pytest.mark.parametrize("name", ["tiny_f32_1k", "zipf_bf16_65k"])
def test_rows_are_unit_norm_in_the_workload_dtype(name):
    w = dataclasses.replace(workloads.WORKLOADS[name], n=min(4096, workloads.WORKLOADS[name].n))
    if w.sizes == "zipf":
        w = dataclasses.replace(w, g=64)
    entries, gid, centres = workloads.make_memory(w, seed=0)
    assert entries.dtype == w.torch_dtype and entries.shape == (w.n, w.d)
    norms = torch.linalg.vector_norm(entries.float(), dim=1)
    tol = 1e-6 if w.dtype == "f32" else 2 ** -7  # bf16 rounding of each coordinate
    assert (norms - 1).abs().max().item() < tol
    assert (centres is None) == (w.embed == "gaussian")


def test_clustered_queries_pick_groups_in_proportion_to_size():
    """A clustered query is its group's centre plus N(0, 0.3^2) noise: the
    nearest centre recovers the group, and groups appear in proportion to
    their sizes (the group of a uniformly drawn entry)."""
    w = dataclasses.replace(workloads.WORKLOADS["zipf_bf16_65k"], n=65536, g=16, d=256, dtype="f32")
    entries, gid, centres = workloads.make_memory(w, seed=0)
    q = workloads.make_queries(w, gid, centres, seed=0, b=20000)
    home = torch.argmax(q @ (centres / torch.linalg.vector_norm(centres, dim=1, keepdim=True)).T, dim=1)
    freq = np.bincount(home.numpy(), minlength=16) / 20000
    sizes = zipf_sizes(65536, 16) / 65536
    np.testing.assert_allclose(freq, sizes, atol=0.012)


def test_append_batches_draw_groups_by_the_initial_weights():
    w = dataclasses.replace(workloads.WORKLOADS["stream_bf16_512k"], n=8192, g=8, d=64, append_per_round=20000)
    _, _, centres = workloads.make_memory(w, seed=0)
    rows, gid = workloads.make_append_batch(w, centres, round_idx=3)
    assert rows.shape == (20000, 64) and rows.dtype == torch.bfloat16 and gid.dtype == torch.int32
    freq = np.bincount(gid.numpy(), minlength=8) / 20000
    np.testing.assert_allclose(freq, zipf_sizes(8192, 8) / 8192, atol=0.012)
    rows2, gid2 = workloads.make_append_batch(w, centres, round_idx=4)
    assert (gid.numpy() != gid2.numpy()).any()
