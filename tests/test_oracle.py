"""Pins for the float64 oracle (CPU only).

Each test ties the oracle to something other than itself: a closed form
worked out from the equations, a library routine that computes the same
quantity a different way (numpy matmul / lexsort, scipy logsumexp), an
invariant the paper's definitions imply, or brute force on a tiny memory.
Together they are chosen so that a plausible slip (a dropped term, a wrong
sign, a transposed operand, a missing 1/n, tau multiplied instead of divided,
a wrong tie order, a leak outside the selected groups) fails at least one.
"""
import math
import os

import numpy as np
import pytest
from scipy.special import logsumexp

import oracle


def _unit_rows(rng, n, d):
    x = rng.standard_normal((n, d))
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    return x.astype(np.float32)


def _bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit pattern with round-to-nearest-even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def _bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------- closed forms

def test_one_hot_memory_by_counting():
    """Entries are unit axis vectors, so a group key's d-th coordinate is the
    fraction of its entries on axis d (the mean, c_g = sum/n_g) and a one-hot
    query e_d scores an entry 1 if it lies on axis d, else 0 (Eq. 9 with the
    linear scorer).  Every expected number below comes from counting."""
    d, n_groups = 4, 3
    gid = np.array([0, 0, 0, 1, 1, 2, 2, 2, 2, 0], dtype=np.int32)
    axis = np.array([0, 1, 0, 2, 2, 3, 1, 3, 3, 3])
    entries = np.zeros((gid.size, d), dtype=np.float32)
    entries[np.arange(gid.size), axis] = 1.0
    cent, counts = oracle.centroids(entries, gid, n_groups)
    for g in range(n_groups):
        members = axis[gid == g]
        for a in range(d):
            assert cent[g, a] == np.count_nonzero(members == a) / members.size
    assert list(counts) == [4, 2, 4]

    for query_axis in range(d):
        q = np.zeros((1, d), dtype=np.float32)
        q[0, query_axis] = 1.0
        frac = [np.count_nonzero(axis[gid == g] == query_axis) / np.count_nonzero(gid == g)
                for g in range(n_groups)]
        want_groups = sorted(range(n_groups), key=lambda g: (-frac[g], g))[:2]
        out = oracle.query(entries, gid, n_groups, q, k_groups=2, k_entries=4, tau=1.0)
        assert list(out["group_idx"][0]) == want_groups
        assert list(out["group_score"][0]) == [frac[g] for g in want_groups]
        cand = [e for e in range(gid.size) if gid[e] in want_groups]
        hit = [e for e in cand if axis[e] == query_axis]
        miss = [e for e in cand if axis[e] != query_axis]
        want_ids = (hit + miss)[:4]          # score 1 before 0, ties to lower id
        assert list(out["entry_idx"][0]) == want_ids
        assert list(out["entry_score"][0]) == [1.0 if axis[e] == query_axis else 0.0 for e in want_ids]
        lse = math.log(len(hit) * math.e + len(miss))
        assert out["lse"][0] == pytest.approx(lse, rel=0, abs=1e-15)
        for e, w in zip(want_ids, out["entry_weight"][0]):
            s = 1.0 if axis[e] == query_axis else 0.0
            assert w == pytest.approx(math.exp(s - lse), rel=1e-15)
        assert out["n_cand"][0] == len(cand)


@pytest.mark.parametrize("tau,eps", [(0.5, 0.0), (0.5, 0.2), (2.0, 0.7)])
def test_two_candidates_closed_form(tau, eps):
    """With two candidates a, b the Eq. 11 mixture is
    w_a = eps/2 + (1-eps) / (1 + exp((s_b - s_a)/tau))."""
    entries = np.array([[0.6, 0.8, 0, 0], [1.0, 0, 0, 0], [0, 0, 1.0, 0]], dtype=np.float32)
    gid = np.array([1, 1, 0], dtype=np.int32)
    q = np.array([[0.28, 0.96, 0, 0]], dtype=np.float32)
    out = oracle.query(entries, gid, 2, q, k_groups=1, k_entries=2, tau=tau, eps=eps)
    assert list(out["group_idx"][0]) == [1]
    s0 = float(np.dot(entries[0].astype(np.float64), q[0].astype(np.float64)))
    s1 = float(np.dot(entries[1].astype(np.float64), q[0].astype(np.float64)))
    assert s0 > s1
    assert list(out["entry_idx"][0]) == [0, 1]
    w0 = eps / 2 + (1 - eps) / (1 + math.exp((s1 - s0) / tau))
    w1 = eps / 2 + (1 - eps) / (1 + math.exp((s0 - s1) / tau))
    assert out["entry_weight"][0][0] == pytest.approx(w0, rel=1e-14)
    assert out["entry_weight"][0][1] == pytest.approx(w1, rel=1e-14)
    assert out["lse"][0] == pytest.approx(math.log(math.exp(s0 / tau) + math.exp(s1 / tau)), rel=1e-14)


def test_single_candidate_has_weight_one():
    entries = np.array([[0.0, 1.0], [1.0, 0.0]], dtype=np.float32)
    gid = np.array([0, 1], dtype=np.int32)
    q = np.array([[0.25, 0.75]], dtype=np.float32)
    out = oracle.query(entries, gid, 2, q, k_groups=1, k_entries=3, tau=0.3, eps=0.5)
    assert list(out["group_idx"][0]) == [0]
    assert list(out["entry_idx"][0]) == [0, -1, -1]
    assert out["entry_weight"][0][0] == pytest.approx(1.0, rel=1e-15)
    assert out["lse"][0] == pytest.approx(0.75 / 0.3, rel=1e-15)
    assert list(out["entry_weight"][0][1:]) == [0.0, 0.0]
    assert np.isneginf(out["entry_score"][0][1:]).all()


def test_cold_softmax_keeps_the_closed_form():
    """Eq. 11 at a temperature where exp(s/tau) overflows a double: scores 0
    and 1 at tau = 1e-3 give lse = 1000 + log(1 + e^-1000) = 1000 and
    weights eps/2 + (1-eps) * {e^-1000, 1}.  The weaker candidate comes first
    in entry order, so the softmax has to shift by the largest s/tau, not by
    whichever candidate it met first."""
    entries = np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0], [0, 0, 1.0, 0]], dtype=np.float32)
    gid = np.array([0, 0, 1], dtype=np.int32)
    q = np.array([[0, 1.0, 0, 0]], dtype=np.float32)
    eps = 0.1
    out = oracle.query(entries, gid, 2, q, k_groups=1, k_entries=2, tau=1e-3, eps=eps)
    assert list(out["group_idx"][0]) == [0]
    assert list(out["entry_idx"][0]) == [1, 0]
    assert out["lse"][0] == pytest.approx(1000.0, rel=1e-15)
    assert out["entry_weight"][0][0] == pytest.approx(eps / 2 + (1 - eps), rel=1e-15)
    assert out["entry_weight"][0][1] == pytest.approx(eps / 2, rel=1e-15)


# ---------------------------------------------------- library-routine special cases

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_all_groups_selected_equals_flat_scan(dtype):
    """k_groups = G selects every non-empty group, so the two-level lookup is
    the flat retrieval of App. C.4 / C.8: a full top-k over all entries, which
    numpy computes independently (matmul + lexsort); lse is scipy's."""
    rng = np.random.default_rng(11)
    n, d, g = 300, 24, 7
    x = _unit_rows(rng, n, d)
    q32 = _unit_rows(rng, 5, d)
    gid = rng.integers(0, g, n).astype(np.int32)
    if dtype == "bf16":
        entries, queries = _bf16_bits(x), _bf16_bits(q32)
        e64, q64 = _bf16_to_f64(entries), _bf16_to_f64(queries)
    else:
        entries, queries = x, q32
        e64, q64 = x.astype(np.float64), q32.astype(np.float64)
    tau = 0.07
    out = oracle.query(entries, gid, g, queries, k_groups=g, k_entries=40, tau=tau, eps=0.0)
    scores = q64 @ e64.T
    for b in range(queries.shape[0]):
        order = np.lexsort((np.arange(n), -scores[b]))[:40]
        assert list(out["entry_idx"][b]) == list(order)
        np.testing.assert_allclose(out["entry_score"][b], scores[b][order], rtol=0, atol=1e-12)
        assert out["lse"][b] == pytest.approx(logsumexp(scores[b] / tau), rel=1e-12)
        np.testing.assert_allclose(out["entry_weight"][b], np.exp(scores[b][order] / tau - logsumexp(scores[b] / tau)),
                                   rtol=1e-11)
        assert out["n_cand"][b] == n


def test_flat_scan_matches_numpy_brute_force():
    """The flat retrieval against numpy: matmul scores, lexsort top-k (ties to
    the lower id, planted by duplicated rows), scipy's logsumexp, and the
    epsilon term of Eq. 11 spread over all n entries."""
    rng = np.random.default_rng(23)
    n, d, b, k, tau, eps = 240, 20, 6, 30, 0.2, 0.15
    x = _unit_rows(rng, n, d)
    x[100:120] = x[0:20]  # equal scores: the lower id must come first
    q = _unit_rows(rng, b, d)
    out = oracle.flat(x, q, k, tau=tau, eps=eps)
    scores = q.astype(np.float64) @ x.astype(np.float64).T
    for r in range(b):
        order = np.lexsort((np.arange(n), -scores[r]))[:k]
        assert list(out["entry_idx"][r]) == list(order)
        np.testing.assert_allclose(out["entry_score"][r], scores[r][order], rtol=0, atol=1e-12)
        lse = logsumexp(scores[r] / tau)
        assert out["lse"][r] == pytest.approx(lse, rel=1e-12)
        np.testing.assert_allclose(out["entry_weight"][r],
                                   eps / n + (1 - eps) * np.exp(scores[r][order] / tau - lse), rtol=1e-11)
        assert out["n_cand"][r] == n
    short = oracle.flat(x[:5], q, 8)
    assert (short["entry_idx"][:, 5:] == -1).all() and (short["entry_weight"][:, 5:] == 0).all()


def test_stage1_matches_numpy_brute_force():
    """Group keys by numpy (bincount means), coarse scores by matmul, top-k by
    lexsort: an independent computation of centroids + stage 1."""
    rng = np.random.default_rng(5)
    n, d, g, kg = 500, 16, 12, 5
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, g, n).astype(np.int32)
    q = _unit_rows(rng, 9, d)
    cent, counts = oracle.centroids(x, gid, g)
    want_counts = np.bincount(gid, minlength=g)
    assert list(counts) == list(want_counts)
    want_cent = np.stack([x[gid == j].astype(np.float64).mean(axis=0) for j in range(g)])
    np.testing.assert_allclose(cent, want_cent, rtol=0, atol=1e-15)
    gi, gs = oracle.stage1(q, cent, counts, kg)
    s1 = q.astype(np.float64) @ want_cent.T
    for b in range(q.shape[0]):
        order = np.lexsort((np.arange(g), -s1[b]))[:kg]
        assert list(gi[b]) == list(order)
        np.testing.assert_allclose(gs[b], s1[b][order], rtol=0, atol=1e-14)


def test_two_level_matches_numpy_brute_force():
    """Whole lookup on a tiny clustered memory against an independent numpy
    brute force (mask by selected groups, lexsort, logsumexp)."""
    rng = np.random.default_rng(7)
    n, d, g, kg, ke = 400, 32, 10, 3, 6
    centres = rng.standard_normal((g, d))
    gid = rng.integers(0, g, n).astype(np.int32)
    x = centres[gid] + 0.3 * rng.standard_normal((n, d))
    x = (x / np.linalg.norm(x, axis=1, keepdims=True)).astype(np.float32)
    q = centres[rng.integers(0, g, 6)] + 0.3 * rng.standard_normal((6, d))
    q = (q / np.linalg.norm(q, axis=1, keepdims=True)).astype(np.float32)
    tau, eps = 0.25, 0.1
    out = oracle.query(x, gid, g, q, kg, ke, tau, eps)
    e64, q64 = x.astype(np.float64), q.astype(np.float64)
    cent = np.stack([e64[gid == j].mean(axis=0) for j in range(g)])
    for b in range(q.shape[0]):
        s1 = cent @ q64[b]
        sel = np.lexsort((np.arange(g), -s1))[:kg]
        mask = np.isin(gid, sel)
        ids = np.nonzero(mask)[0]
        s2 = e64[ids] @ q64[b]
        order = np.lexsort((ids, -s2))[:ke]
        lse = logsumexp(s2 / tau)
        assert list(out["group_idx"][b]) == list(sel)
        assert list(out["entry_idx"][b]) == list(ids[order])
        np.testing.assert_allclose(out["entry_score"][b], s2[order], atol=1e-13, rtol=0)
        np.testing.assert_allclose(out["entry_weight"][b],
                                   eps / ids.size + (1 - eps) * np.exp(s2[order] / tau - lse), rtol=1e-11)
        assert out["lse"][b] == pytest.approx(lse, rel=1e-13)


# ------------------------------------------------------------------ invariants

@pytest.mark.parametrize("tau,eps", [(1.0, 0.0), (0.05, 0.0), (1.0, 0.1), (0.3, 1.0)])
def test_weights_over_full_candidate_set_sum_to_one(tau, eps):
    rng = np.random.default_rng(3)
    n, d, g = 200, 8, 6
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, g, n).astype(np.int32)
    q = _unit_rows(rng, 4, d)
    out = oracle.query(x, gid, g, q, k_groups=3, k_entries=n, tau=tau, eps=eps)
    for b in range(4):
        nb = out["n_cand"][b]
        w = out["entry_weight"][b][:nb]
        assert math.fsum(w) == pytest.approx(1.0, abs=1e-12)
        assert (out["entry_idx"][b][nb:] == -1).all()
        if eps == 1.0:
            np.testing.assert_allclose(w, 1.0 / nb, rtol=1e-15)


def test_restriction_to_selected_groups():
    """Eq. 12: every returned entry belongs to a selected group, and the
    candidate count is the selected groups' total size."""
    rng = np.random.default_rng(9)
    n, d, g = 1000, 16, 20
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, g, n).astype(np.int32)
    q = _unit_rows(rng, 12, d)
    out = oracle.query(x, gid, g, q, k_groups=4, k_entries=25)
    counts = np.bincount(gid, minlength=g)
    for b in range(12):
        sel = set(out["group_idx"][b])
        assert all(gid[e] in sel for e in out["entry_idx"][b])
        assert out["n_cand"][b] == sum(counts[s] for s in sel)


def test_entry_permutation_only_relabels():
    rng = np.random.default_rng(2)
    n, d, g = 256, 12, 8
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, g, n).astype(np.int32)
    q = _unit_rows(rng, 5, d)
    perm = rng.permutation(n)
    a = oracle.query(x, gid, g, q, 3, 10)
    b = oracle.query(x[perm], gid[perm], g, q, 3, 10)
    assert (a["group_idx"] == b["group_idx"]).all()
    np.testing.assert_array_equal(a["entry_idx"], perm[b["entry_idx"]])
    np.testing.assert_array_equal(a["entry_score"], b["entry_score"])
    np.testing.assert_allclose(a["lse"], b["lse"], rtol=1e-14)


def test_empty_groups_never_selected_and_padding():
    rng = np.random.default_rng(4)
    d, g = 8, 8
    gid = np.array([0, 2, 3, 4, 6, 7] * 5, dtype=np.int32)  # groups 1 and 5 empty
    x = _unit_rows(rng, gid.size, d)
    q = _unit_rows(rng, 3, d)
    out = oracle.query(x, gid, g, q, k_groups=8, k_entries=gid.size + 5)
    for b in range(3):
        assert sorted(out["group_idx"][b][:6]) == [0, 2, 3, 4, 6, 7]
        assert list(out["group_idx"][b][6:]) == [-1, -1]
        assert np.isneginf(out["group_score"][b][6:]).all()
        assert list(out["entry_idx"][b][-5:]) == [-1] * 5
        assert (out["entry_weight"][b][-5:] == 0).all()


def test_ties_go_to_lower_index():
    d = 4
    row = np.array([0.5, 0.5, 0.5, 0.5], dtype=np.float32)
    other = np.array([1.0, 0, 0, 0], dtype=np.float32)
    # groups 0 and 2 hold identical rows (equal keys and scores), group 1 differs
    entries = np.stack([row, other, row, row, other, row])
    gid = np.array([2, 1, 0, 2, 1, 0], dtype=np.int32)
    q = np.array([[0.5, 0.5, 0.5, 0.5]], dtype=np.float32)
    out = oracle.query(entries, gid, 3, q, k_groups=2, k_entries=4)
    assert list(out["group_idx"][0]) == [0, 2]
    assert out["group_score"][0][0] == out["group_score"][0][1]
    assert list(out["entry_idx"][0]) == [0, 2, 3, 5]


def test_tau_changes_weights_not_ranking():
    rng = np.random.default_rng(8)
    x = _unit_rows(rng, 300, 16)
    gid = rng.integers(0, 6, 300).astype(np.int32)
    q = _unit_rows(rng, 4, 16)
    base = oracle.query(x, gid, 6, q, 2, 12, tau=1.0)
    for tau in (0.05, 20.0):
        out = oracle.query(x, gid, 6, q, 2, 12, tau=tau)
        np.testing.assert_array_equal(out["entry_idx"], base["entry_idx"])
        assert (np.diff(out["entry_weight"], axis=1) <= 0).all()
    flat = oracle.query(x, gid, 6, q, 2, 12, tau=1e7)
    for b in range(4):
        np.testing.assert_allclose(flat["entry_weight"][b], 1.0 / flat["n_cand"][b], rtol=1e-6)


def test_query_scale_doubles_scores_exactly():
    rng = np.random.default_rng(6)
    x = _unit_rows(rng, 100, 8)
    gid = rng.integers(0, 4, 100).astype(np.int32)
    q = _unit_rows(rng, 3, 8)
    a = oracle.query(x, gid, 4, q, 2, 5)
    b = oracle.query(x, gid, 4, 2 * q, 2, 5)
    np.testing.assert_array_equal(b["entry_idx"], a["entry_idx"])
    np.testing.assert_array_equal(b["entry_score"], 2 * a["entry_score"])
    np.testing.assert_array_equal(b["group_score"], 2 * a["group_score"])


def test_bf16_bits_read_exactly():
    rng = np.random.default_rng(1)
    bits = _bf16_bits(_unit_rows(rng, 64, 16))
    qbits = _bf16_bits(_unit_rows(rng, 2, 16))
    gid = rng.integers(0, 4, 64).astype(np.int32)
    a = oracle.query(bits, gid, 4, qbits, 2, 8)
    b = oracle.query(_bf16_to_f64(bits).astype(np.float32), gid, 4,
                     _bf16_to_f64(qbits).astype(np.float32), 2, 8)
    for k in ("group_idx", "entry_idx", "entry_score", "entry_weight", "lse"):
        np.testing.assert_array_equal(a[k], b[k])


def test_centroid_chunks_and_incremental_mean():
    """Feeding entries in chunks gives the same sums; the mean after an
    append equals (n_g c_g + sum of new rows) / (n_g + m_g), the in-place
    update rule the CUDA path uses for Eq. 15."""
    rng = np.random.default_rng(12)
    x = _unit_rows(rng, 90, 8)
    gid = rng.integers(0, 5, 90).astype(np.int32)
    whole, counts = oracle.centroids(x, gid, 5)
    acc = oracle.CentroidAccumulator(5, 8)
    for s in range(0, 90, 40):
        acc.add(x[s:s + 40], gid[s:s + 40])
    chunked, counts2 = acc.finalize()
    np.testing.assert_array_equal(chunked, whole)
    old, old_n = oracle.centroids(x[:60], gid[:60], 5)
    new_sum = np.zeros((5, 8))
    np.add.at(new_sum, gid[60:], x[60:].astype(np.float64))
    new_n = np.bincount(gid[60:], minlength=5)
    inc = (old * old_n[:, None] + new_sum) / (old_n + new_n)[:, None]
    np.testing.assert_allclose(inc, whole, rtol=1e-14, atol=1e-15)


def test_bad_group_id_rejected():
    x = np.zeros((3, 8), dtype=np.float32)
    with pytest.raises(ValueError):
        oracle.centroids(x, np.array([0, 5, 1], dtype=np.int32), 3)


# ------------------------------------------------ prefix-attended query (N1)

def test_prefix_of_one_is_the_query():
    """A prefix of length 1 has the single weight exp(0) = 1, so the reduced
    query is the query itself, for any lambda."""
    rng = np.random.default_rng(11)
    q = _unit_rows(rng, 6, 32)[:, None, :]
    for lam in (0.0, 0.5, 3.0):
        assert np.array_equal(oracle.prefix_reduce(q, lam), q[:, 0, :].astype(np.float64))


@pytest.mark.parametrize("lam", [0.0, 0.5, 1.7])
def test_prefix_weights_newest_one_and_geometric(lam):
    """With q_i the i-th unit axis vector, coordinate i of the reduced query is
    alpha_i: the newest element (i = P) weighs exactly 1, and each older one
    weighs exp(-lambda) times the next (Eq. 10); lambda = 0 weighs all ones."""
    P = 7
    q = np.eye(P, 10, dtype=np.float32)[None, :, :]
    a = oracle.prefix_reduce(q, lam)[0]
    assert a[P - 1] == 1.0
    for i in range(P - 1):
        assert a[i] == pytest.approx(a[i + 1] * math.exp(-lam), rel=1e-14)
    assert np.all(a[P:] == 0.0)


@pytest.mark.parametrize("lam,P", [(0.0, 5), (0.5, 6), (2.0, 3)])
def test_constant_prefix_sums_a_geometric_series(lam, P):
    """P copies of one query reduce to that query times sum_{m=0}^{P-1}
    exp(-lambda m) = (1 - exp(-lambda P)) / (1 - exp(-lambda)) (P at lambda = 0)."""
    rng = np.random.default_rng(12)
    q = _unit_rows(rng, 3, 16)
    prefix = np.repeat(q[:, None, :], P, axis=1)
    total = P if lam == 0.0 else (1.0 - math.exp(-lam * P)) / (1.0 - math.exp(-lam))
    np.testing.assert_allclose(oracle.prefix_reduce(prefix, lam), q.astype(np.float64) * total,
                               rtol=1e-13, atol=0)


def test_prefix_scores_are_weighted_stage1_scores():
    """Eq. 9 summed over the prefix: the group scores of the reduced query are
    the alpha-weighted sums of the group scores of the prefix elements, each
    scored on its own by stage 1 (linearity of the scorer)."""
    rng = np.random.default_rng(13)
    G, d, P, lam = 12, 24, 5, 0.7
    entries = _unit_rows(rng, 300, d)
    gid = rng.integers(0, G, 300).astype(np.int32)
    cent, counts = oracle.centroids(entries, gid, G)
    prefix = _unit_rows(rng, 4 * P, d).reshape(4, P, d)
    alpha = np.empty(P)
    alpha[P - 1] = 1.0
    for i in range(P - 2, -1, -1):
        alpha[i] = alpha[i + 1] * math.exp(-lam)

    def all_scores(qs):
        gi, gs = oracle.stage1(qs, cent, counts, G)
        out = np.empty((qs.shape[0], G))
        for b in range(qs.shape[0]):
            out[b, gi[b]] = gs[b]
        return out

    per_elem = np.stack([all_scores(np.ascontiguousarray(prefix[:, i, :])) for i in range(P)], axis=1)
    want = np.einsum("i,big->bg", alpha, per_elem)
    got = all_scores(oracle.round_query(oracle.prefix_reduce(prefix, lam), "f32"))
    np.testing.assert_allclose(got, want, rtol=0, atol=2e-6)


def test_round_query_bf16_is_round_to_nearest_even():
    """The reduced query is rounded to bf16 the way any bf16 query is made:
    float64 -> float32 -> bf16, each step to nearest, ties to even.  Checked
    against torch's float32 -> bfloat16 conversion (an independent library
    routine) on random values over many binades, and on hand-made float32
    patterns whose dropped half is exactly 0x8000 (a tie: even lsb stays,
    odd lsb rounds up), just below and just above it, and carries that ripple
    into the exponent."""
    import torch

    rng = np.random.default_rng(41)
    x = rng.standard_normal(20000) * np.exp2(rng.integers(-30, 30, 20000))
    got = oracle.round_query(x, "bf16")
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, want)
    cases = {
        0x3F808000: 0x3F80,  # tie, even lsb: stays
        0x3F818000: 0x3F82,  # tie, odd lsb: up to even
        0x3F807FFF: 0x3F80,  # just below the half: down
        0x3F808001: 0x3F81,  # just above the half: up
        0xBF818000: 0xBF82,  # negative tie, odd lsb: magnitude up
        0x3F7FFFFF: 0x3F80,  # carry into the exponent
        0x00008000: 0x0000,  # subnormal tie, even lsb
        0x00018000: 0x0002,  # subnormal tie, odd lsb
    }
    bits = np.array(list(cases), dtype=np.uint32)
    got = oracle.round_query(bits.view(np.float32).astype(np.float64), "bf16")
    assert [int(v) for v in got] == list(cases.values())
    # The float64 -> float32 step rounds to nearest too: a double just above
    # the float32 midpoint of 1 and 1 + 2^-23 goes up, bf16 then keeps 1.0.
    assert oracle.round_query(np.array([1.0 + 2.0 ** -24 + 2.0 ** -40]), "f32").view(np.uint32)[0] == 0x3F800001


# ------------------------------------------------ edge-table routing (N2)

def test_edge_scores_one_hot_weights_read_the_feature_slice():
    """With w the f-th unit vector and a one-element prefix (weight 1), the
    score of g is the f-th feature of the edge from the prefix group to g:
    Z[p, g, f] (row = from, column = to)."""
    rng = np.random.default_rng(21)
    G, F = 7, 4
    Z = rng.standard_normal((G, G, F)).astype(np.float32)
    prefix = np.array([[3], [0], [6]], dtype=np.int32)
    for f in range(F):
        w = np.zeros(F)
        w[f] = 1.0
        s = oracle.edge_scores(Z, w, prefix, 0.8)
        for b, p in enumerate(prefix[:, 0]):
            assert np.array_equal(s[b], Z[p, :, f].astype(np.float64))


def test_edge_scores_linear_in_weights():
    rng = np.random.default_rng(22)
    G, F = 9, 12
    Z = rng.standard_normal((G, G, F)).astype(np.float32)
    prefix = rng.integers(-1, G, (5, 4)).astype(np.int32)
    w1, w2 = rng.standard_normal(F), rng.standard_normal(F)
    np.testing.assert_allclose(oracle.edge_scores(Z, w1 + w2, prefix, 0.3),
                               oracle.edge_scores(Z, w1, prefix, 0.3) + oracle.edge_scores(Z, w2, prefix, 0.3),
                               rtol=0, atol=1e-12)


@pytest.mark.parametrize("lam", [0.0, 0.6])
def test_edge_prefix_weights_newest_one_and_geometric(lam):
    """Z has a 1 on every edge leaving group k (feature 0) and 0 elsewhere, so
    a prefix holding k at one position and nothing (-1) elsewhere scores every
    group with that position's weight (Eq. 10): 1 for the newest, e^{-lambda}
    times the next one for each older; an empty prefix scores 0."""
    G, F, P, k = 6, 2, 5, 4
    Z = np.zeros((G, G, F), dtype=np.float32)
    Z[k, :, 0] = 1.0
    w = np.array([1.0, 0.0])
    prefix = np.full((P + 1, P), -1, dtype=np.int32)
    for i in range(P):
        prefix[i, i] = k
    s = oracle.edge_scores(Z, w, prefix, lam)
    assert np.all(s[P - 1] == 1.0)
    for i in range(P - 1):
        np.testing.assert_allclose(s[i], s[i + 1] * math.exp(-lam), rtol=1e-14)
    assert np.all(s[P] == 0.0)


def test_select_matches_lexsort_without_empty_groups():
    rng = np.random.default_rng(23)
    b, G, k = 6, 30, 8
    scores = np.round(rng.standard_normal((b, G)), 1)       # many ties
    counts = rng.integers(0, 3, G)
    gi, gs = oracle.select(scores, counts, k)
    for q in range(b):
        live = np.nonzero(counts > 0)[0]
        order = live[np.lexsort((live, -scores[q, live]))][:k]
        assert list(gi[q, :len(order)]) == list(order)
        assert np.all(gi[q, len(order):] == -1)
        np.testing.assert_array_equal(gs[q, :len(order)], scores[q, order])


# ------------------------------------------- sampling from the policy (Eq. 11)

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def test_philox_known_answers():
    """Philox4x32-10 against the published known-answer vectors."""
    n = 0
    for line in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")):
        words = line.split("#")[0].split()
        if not words:
            continue
        v = [int(x, 16) for x in words]
        assert list(oracle.philox4x32_10(v[0:4], v[4:6])) == v[6:10]
        n += 1
    assert n == 3


def test_policy_uniforms_are_uniform_and_uncorrelated():
    """Kolmogorov-Smirnov against U(0, 1); neighbouring groups (words of one
    generator call) and neighbouring queries are uncorrelated; the seed and
    the offset change the stream."""
    from scipy import stats

    u = np.array([[oracle.policy_uniform(7, 3, b, g) for g in range(64)] for b in range(400)])
    assert (u > 0).all() and (u < 1).all()
    assert stats.kstest(u.ravel(), "uniform").pvalue > 1e-4
    assert abs(np.corrcoef(u[:, :-1].ravel(), u[:, 1:].ravel())[0, 1]) < 0.02
    assert abs(np.corrcoef(u[:-1].ravel(), u[1:].ravel())[0, 1]) < 0.02
    assert oracle.policy_uniform(8, 3, 0, 0) != u[0, 0]
    assert oracle.policy_uniform(7, 4, 0, 0) != u[0, 0]
    assert oracle.policy_uniform(7, 3 + (1 << 32), 0, 0) != u[0, 0]


def _policy_case(B, eps, tau, seed=11):
    scores = np.tile(np.array([0.3, -0.2, 0.9, 0.1, 0.5, 0.0]), (B, 1))
    counts = np.array([3, 2, 4, 0, 1, 5], dtype=np.int64)
    keys, mu = oracle.policy_keys(scores, counts, tau, eps, seed, 0)
    ne = counts > 0
    from scipy.special import softmax

    p = np.zeros(6)
    p[ne] = eps / ne.sum() + (1 - eps) * softmax(scores[0][ne] / tau)
    return scores, counts, keys, mu, p


@pytest.mark.parametrize("eps,tau", [(0.2, 0.4), (0.0, 1.0), (1.0, 0.3)])
def test_first_draw_follows_the_policy(eps, tau):
    """mu equals Eq. 11 by scipy's softmax over the non-empty groups, and the
    group with the largest key (the first draw) has that distribution
    (chi-square over 40,000 independent queries); the empty group never."""
    from scipy import stats

    B = 40000
    _, counts, keys, mu, p = _policy_case(B, eps, tau)
    np.testing.assert_allclose(mu[0], p, rtol=1e-12, atol=0)
    first = keys.argmax(axis=1)
    obs = np.bincount(first, minlength=6)
    assert obs[3] == 0
    ne = counts > 0
    assert stats.chisquare(obs[ne], B * p[ne]).pvalue > 1e-4


def test_second_draw_is_without_replacement():
    """The second-largest key follows P(second = j) = sum_{i != j} p_i p_j / (1 - p_i),
    the law of a second draw without replacement."""
    from scipy import stats

    B = 40000
    _, counts, keys, mu, p = _policy_case(B, 0.1, 0.5, seed=5)
    order = np.argsort(-keys, axis=1, kind="stable")
    assert (order[:, 0] != order[:, 1]).all()
    q = np.array([sum(p[i] * p[j] / (1 - p[i]) for i in range(6) if i != j and p[i] > 0) for j in range(6)])
    np.testing.assert_allclose(q.sum(), 1.0, rtol=1e-12)
    obs = np.bincount(order[:, 1], minlength=6)
    ne = counts > 0
    assert obs[3] == 0
    assert stats.chisquare(obs[ne], B * q[ne]).pvalue > 1e-4


def test_cold_policy_draws_the_top_groups():
    """With a tiny temperature and no exploration the noise cannot reorder
    groups whose scores differ by much more than tau, so the draws are
    stage 1's ranking."""
    rng = np.random.default_rng(9)
    B, G, k = 50, 40, 6
    scores = rng.permutation(G)[None, :].repeat(B, 0) * 0.1 + rng.standard_normal((B, 1))
    counts = np.ones(G, dtype=np.int64)
    counts[[3, 17]] = 0
    keys, _ = oracle.policy_keys(scores, counts, 1e-3, 0.0, 3, 1)
    gi, _ = oracle.select(keys, counts, k)
    ref, _ = oracle.select(scores, counts, k)
    assert (gi == ref).all()


def test_policy_rows_keep_their_query_uniforms():
    """A sample of a batch's rows, passed with their query ids, draws what
    the whole batch draws for those rows."""
    rng = np.random.default_rng(4)
    scores = rng.standard_normal((30, 12))
    counts = np.arange(12, dtype=np.int64) % 5
    full, _ = oracle.policy_keys(scores, counts, 0.7, 0.1, 99, 7)
    rows = np.array([29, 3, 17])
    part, _ = oracle.policy_keys(scores[rows], counts, 0.7, 0.1, 99, 7, query_ids=rows)
    np.testing.assert_array_equal(part, full[rows])
    other, _ = oracle.policy_keys(scores[rows], counts, 0.7, 0.1, 99, 7)
    assert not np.array_equal(other, full[rows])


# ------------------------------------------------ nearest-key append (Eq. 15)

def test_assign_nearest_matches_numpy_brute_force():
    """Entries appended without a group join the non-empty group whose key
    scores highest (numpy argmax with lexsort ties; duplicated keys force
    ties to the lower id); given ids are kept."""
    rng = np.random.default_rng(31)
    d, G = 16, 9
    keys = _unit_rows(rng, G, d).astype(np.float64)
    keys[5] = keys[2]  # a tie: group 2 must win
    counts = np.array([3, 0, 2, 1, 4, 2, 5, 0, 1], dtype=np.int64)
    x = _unit_rows(rng, 200, d)
    x[:10] = keys[2].astype(np.float32)  # rows that tie between groups 2 and 5
    gid = np.where(rng.random(200) < 0.6, -1, rng.integers(0, G, 200)).astype(np.int32)
    gid[:10] = -1
    out = oracle.assign_nearest(x, gid, keys, counts)
    s = x.astype(np.float64) @ keys.T
    s[:, counts == 0] = -np.inf
    for i in range(200):
        if gid[i] >= 0:
            assert out[i] == gid[i]
        else:
            assert out[i] == np.lexsort((np.arange(G), -s[i]))[0]
    assert (out[:10] == 2).all()
    assert not np.isin(out[gid == -1], [1, 7]).any()


# ------------------------------------------------ composed lookups (N2, N4)

def _brute_stage2(x, gid, q, groups, k, tau, eps):
    """Stage 2 written out with numpy: candidates = entries of `groups`,
    matmul scores, lexsort top-k (ties to the lower id), scipy logsumexp."""
    cand = np.flatnonzero(np.isin(gid, groups))
    s = x[cand].astype(np.float64) @ q.astype(np.float64)
    order = np.lexsort((cand, -s))[:k]
    lse = logsumexp(s / tau)
    w = eps / cand.size + (1 - eps) * np.exp(s[order] / tau - lse)
    return cand[order], s[order], w, lse


def test_edge_routed_lookup_by_inspection():
    """One feature, w = 1 and Z[p, g] = -(g - p)^2: a query whose prefix is
    the single group p ranks p first, then its neighbours by distance, the
    lower id first on ties, skipping empty groups (3 here).  The group
    scores are -(g - p)^2 exactly (a one-element prefix weighs 1), and the
    entries are the brute-force stage 2 over exactly those groups."""
    G, d, n, kg, ke, tau, eps = 10, 8, 500, 4, 6, 0.7, 0.1
    rng = np.random.default_rng(43)
    Z = np.zeros((G, G, 1), np.float32)
    for p in range(G):
        for g in range(G):
            Z[p, g, 0] = -float((g - p) ** 2)
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, G, n).astype(np.int32)
    gid[gid == 3] = 2
    prefix = np.array([[5], [0], [9]], np.int32)
    q = _unit_rows(rng, 3, d)
    out = oracle.query_edges(x, gid, G, Z, np.array([1.0]), prefix, 0.5, q, kg, ke, tau=tau, eps=eps)
    want = [[5, 4, 6, 7], [0, 1, 2, 4], [9, 8, 7, 6]]
    for r, p in enumerate(prefix[:, 0]):
        assert list(out["group_idx"][r]) == want[r]
        assert list(out["group_score"][r]) == [-float((g - p) ** 2) for g in want[r]]
        ids, s, w, lse = _brute_stage2(x, gid, q[r], want[r], ke, tau, eps)
        assert list(out["entry_idx"][r]) == list(ids)
        np.testing.assert_allclose(out["entry_score"][r], s, rtol=0, atol=1e-12)
        np.testing.assert_allclose(out["entry_weight"][r], w, rtol=1e-11)
        assert out["lse"][r] == pytest.approx(lse, rel=1e-12)


def test_sampled_lookup_cold_limit_is_the_ranked_lookup():
    """As tau -> 0 the policy of Eq. 11 puts all its mass on the best group:
    with score gaps of at least 5e-3 and tau = 1e-4, log-probability gaps
    (>= 50) exceed any Gumbel spread (about 20 for 23-bit uniforms).  So the
    draws are stage 1's ranking, and the sampled lookup returns the ranked
    lookup's groups, entries, weights and lse, for every seed."""
    rng = np.random.default_rng(44)
    n, d, G, b, kg, ke, tau = 600, 12, 10, 8, 3, 7, 1e-4
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, G, n).astype(np.int32)
    cent, counts = oracle.centroids(x, gid, G)
    q = _unit_rows(rng, 64, d)
    s = -np.sort(-(q.astype(np.float64) @ cent.T), axis=1)
    gaps = (s[:, :kg] - s[:, 1:kg + 1]).min(axis=1)
    q = q[gaps > 5e-3][:b]
    assert q.shape[0] == b
    ref = oracle.query(x, gid, G, q, kg, ke, tau=tau)
    for seed in (0, 1, 7):
        out = oracle.query_sampled(x, gid, G, q, kg, ke, tau, 0.0, seed, 3, centroid=cent, counts=counts)
        assert np.array_equal(out["group_idx"], ref["group_idx"])
        assert np.array_equal(out["entry_idx"], ref["entry_idx"])
        np.testing.assert_allclose(out["entry_weight"], ref["entry_weight"], rtol=1e-12)
        np.testing.assert_allclose(out["lse"], ref["lse"], rtol=1e-12)


def test_sampled_lookup_draws_uniformly_at_full_exploration():
    """With eps = 1 the policy of Eq. 11 is uniform over the non-empty groups,
    whatever the scores: over many seeds the sampled lookup's first group is
    uniform (chi-square), its groups are distinct and never empty, and its
    entries are the brute-force stage 2 over the drawn groups."""
    from scipy.stats import chisquare

    rng = np.random.default_rng(45)
    n, d, G, kg, ke = 300, 8, 6, 2, 5
    x = _unit_rows(rng, n, d)
    gid = rng.integers(0, G, n).astype(np.int32)
    gid[gid == 4] = 5  # group 4 empty
    q = _unit_rows(rng, 1, d)
    cent, counts = oracle.centroids(x, gid, G)
    first = []
    for seed in range(1500):
        out = oracle.query_sampled(x, gid, G, q, kg, ke, 0.5, 1.0, seed, 0, centroid=cent, counts=counts)
        gi = out["group_idx"][0]
        assert len(set(gi.tolist())) == kg and 4 not in gi and (gi >= 0).all()
        if seed < 20:
            ids, s, w, lse = _brute_stage2(x, gid, q[0], gi, ke, 0.5, 1.0)
            assert list(out["entry_idx"][0]) == list(ids)
            np.testing.assert_allclose(out["entry_weight"][0], w, rtol=1e-11)
        first.append(gi[0])
    obs = np.bincount(first, minlength=G)[[0, 1, 2, 3, 5]]
    assert chisquare(obs).pvalue > 1e-3
