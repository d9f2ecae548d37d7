"""GPU-vs-oracle comparison rules shared by the parity tests.

Index rule: with t_k and t_{k+1} the oracle's k-th and (k+1)-th scores, the
returned set must equal the oracle's when t_k - t_{k+1} > 1e-3; otherwise every
oracle index scoring above t_k + 1e-3 must be returned and every returned
index must score at least t_k - 1e-3 (exact oracle scores).  The order must
agree wherever adjacent scores differ by more than 1e-3.  Padding (-1) must
match exactly.

Value rule: |gpu - ref| <= rtol * |ref| + atol with (rtol, atol) =
(2e-2, 1e-4) for bf16 inputs and (1e-5, 1e-7) for fp32 inputs.
"""
from __future__ import annotations

import numpy as np

GAP = 1e-3
TOL = {"bf16": (2e-2, 1e-4), "f32": (1e-5, 1e-7)}


def close(gpu, ref, dtype) -> bool:
    rtol, atol = TOL[dtype]
    gpu, ref = float(gpu), float(ref)
    if np.isneginf(ref):
        return np.isneginf(gpu)
    return abs(gpu - ref) <= rtol * abs(ref) + atol


def check_ranked(what, gpu_ids, gpu_scores, ref_ids, ref_scores, k, exact_score, dtype, tol=None):
    """gpu_ids/gpu_scores: length k.  ref_ids/ref_scores: the oracle's ranking
    of length >= k+1 (padded with -1 / -inf).  exact_score(id) gives the
    oracle's (float64) score of any id.  tol(id), when given, replaces the
    dtype's value tolerance with an absolute bound.  Returns a list of problems."""
    bad = []
    gpu_ids = [int(x) for x in gpu_ids[:k]]
    ref_ids = [int(x) for x in ref_ids]
    v_ref = sum(1 for x in ref_ids[:k] if x >= 0)
    v_gpu = sum(1 for x in gpu_ids if x >= 0)
    if v_ref != v_gpu or any(x < 0 for x in gpu_ids[:v_gpu]) or any(x >= 0 for x in gpu_ids[v_gpu:]):
        return [f"{what}: padding differs (gpu {gpu_ids}, oracle {ref_ids[:k]})"]
    if len(set(gpu_ids[:v_gpu])) != v_gpu:
        return [f"{what}: duplicate ids {gpu_ids}"]
    if v_ref < k:
        if set(gpu_ids[:v_gpu]) != set(ref_ids[:v_ref]):
            bad.append(f"{what}: candidate set differs")
    else:
        t_k = float(ref_scores[k - 1])
        t_next = float(ref_scores[k]) if len(ref_scores) > k else -np.inf
        if t_k - t_next > GAP:
            if set(gpu_ids) != set(ref_ids[:k]):
                bad.append(f"{what}: set differs with a clear gap ({t_k - t_next:.3g}): "
                           f"gpu {sorted(set(gpu_ids) - set(ref_ids[:k]))} oracle {sorted(set(ref_ids[:k]) - set(gpu_ids))}")
        else:
            must = {ref_ids[i] for i in range(k) if float(ref_scores[i]) > t_k + GAP}
            if not must <= set(gpu_ids):
                bad.append(f"{what}: missing clearly-better ids {sorted(must - set(gpu_ids))}")
            for x in gpu_ids:
                if exact_score(x) < t_k - GAP:
                    bad.append(f"{what}: id {x} scores {exact_score(x):.6g} < t_k - gap ({t_k:.6g})")
    es = [exact_score(x) for x in gpu_ids[:v_gpu]]
    run_min = np.inf
    for i in range(v_gpu):
        if es[i] > run_min + GAP:
            bad.append(f"{what}: order differs at position {i}")
            break
        run_min = min(run_min, es[i])
    for i in range(v_gpu):
        ok = abs(float(gpu_scores[i]) - es[i]) <= tol(gpu_ids[i]) if tol else close(gpu_scores[i], es[i], dtype)
        if not ok:
            bad.append(f"{what}: score of id {gpu_ids[i]} gpu {float(gpu_scores[i]):.7g} oracle {es[i]:.7g}")
            break
    return bad


def compare_lookup(out, entries_np, gid_np, n_groups, queries_np, k_groups, k_entries, tau, eps, dtype,
                   rows=None, centroid=None, counts=None, nthreads=None):
    """Checks the GPU outputs of the queries listed in `rows` (all by default)
    against the oracle: stage 1 directly, stage 2 given the groups the GPU
    selected (so that a near-tie at the group level cannot cascade)."""
    import oracle

    gi = out["group_idx"].cpu().numpy()
    gs = out["group_score"].cpu().numpy()
    ei = out["entry_idx"].cpu().numpy()
    es = out["entry_score"].cpu().numpy()
    ew = out["entry_weight"].cpu().numpy()
    lse = out["lse"].cpu().numpy()
    B = queries_np.shape[0]
    rows = np.arange(B) if rows is None else np.asarray(rows)
    q = queries_np[rows]
    if centroid is None:
        centroid, counts = oracle.centroids(entries_np, gid_np, n_groups, nthreads)
    ref_gi, ref_gs = oracle.stage1(q, centroid, counts, min(k_groups + 1, n_groups), nthreads)
    if ref_gi.shape[1] == k_groups:  # k_groups == n_groups: pad the (k+1)-th
        ref_gi = np.concatenate([ref_gi, -np.ones((len(rows), 1), np.int32)], axis=1)
        ref_gs = np.concatenate([ref_gs, np.full((len(rows), 1), -np.inf)], axis=1)
    n_extra = 16
    ref2 = oracle.stage2(entries_np, gid_np, n_groups, q, gi[rows], k_entries + n_extra, tau, eps, nthreads)
    qf = _as_f64(q)
    problems = []
    for r, b in enumerate(rows):
        cent_score = lambda g, r=r: float(centroid[g] @ qf[r])
        problems += check_ranked(f"query {b} groups", gi[b], gs[b], ref_gi[r], ref_gs[r], k_groups,
                                 cent_score, dtype)
        problems += _check_entries(ei, es, ew, lse, b, r, ref2, entries_np, qf, k_entries, tau, eps, dtype)
    return problems


def _check_entries(ei, es, ew, lse, b, r, ref2, entries_np, qf, k_entries, tau, eps, dtype):
    """Stage 2 of query b (row r of the oracle's stage-2 results)."""
    problems = []
    ref_map = {int(i): (float(s), float(w)) for i, s, w in
               zip(ref2["entry_idx"][r], ref2["entry_score"][r], ref2["entry_weight"][r]) if i >= 0}

    def entry_score(e, r=r):
        if e in ref_map:
            return ref_map[e][0]
        return float(_as_f64(entries_np[e:e + 1])[0] @ qf[r])

    problems += check_ranked(f"query {b} entries", ei[b], es[b], ref2["entry_idx"][r],
                             ref2["entry_score"][r], k_entries, entry_score, dtype)
    nb = int(ref2["n_cand"][r])
    for i in range(k_entries):
        e = int(ei[b][i])
        if e < 0:
            if ew[b][i] != 0:
                problems.append(f"query {b}: padded weight not 0")
            continue
        s_ref = entry_score(e)
        w_ref = ref_map[e][1] if e in ref_map else eps / nb + (1 - eps) * np.exp(s_ref / tau - ref2["lse"][r])
        if not close(ew[b][i], w_ref, dtype):
            problems.append(f"query {b}: weight of id {e} gpu {ew[b][i]:.7g} oracle {w_ref:.7g}")
            break
    if not close(lse[b], ref2["lse"][r], dtype):
        problems.append(f"query {b}: lse gpu {lse[b]:.7g} oracle {ref2['lse'][r]:.7g}")
    return problems


def edge_score_tol(scores, mag, n_features, p_len):
    """Absolute bounds for the fp32 edge-table scores of Eq. 9 (App. B.6
    utility): the fp32 value gate 1e-5 |ref| + 1e-7 wherever the sum is well
    conditioned, widened where it cancels to the textbook bound of an fp32
    sum of n rounded terms, gamma_n * sum |terms| with gamma_n = n u / (1 - n u)
    and u = 2^-24 (Higham, Accuracy and Stability of Numerical Algorithms,
    §3.1).  The kernels take, per prefix element, n_features fused
    multiply-adds for w . z, then one more to add alpha_i times it, and alpha_i
    is rounded once to fp32: n = n_features + p_len + 1.  mag is the oracle's
    score with |Z| and |w|, i.e. sum_i alpha_i sum_f |w_f| |Z_f|."""
    rtol, atol = TOL["f32"]
    n = n_features + p_len + 1
    u = 2.0 ** -24
    gamma = n * u / (1.0 - n * u)
    return np.maximum(rtol * np.abs(np.asarray(scores, dtype=np.float64)) + atol,
                      gamma * np.asarray(mag, dtype=np.float64))


def compare_edge_lookup(out, entries_np, gid_np, n_groups, Z, w, prefix, lam, queries_np, k_groups, k_entries,
                        tau, eps, dtype, nthreads=None):
    """The edge-routed lookup: stage 1 against the oracle's edge-table scores
    (values within edge_score_tol), stage 2 given the GPU's groups."""
    import oracle

    gi = out["group_idx"].cpu().numpy()
    gs = out["group_score"].cpu().numpy()
    ei = out["entry_idx"].cpu().numpy()
    es = out["entry_score"].cpu().numpy()
    ew = out["entry_weight"].cpu().numpy()
    lse = out["lse"].cpu().numpy()
    counts = np.bincount(np.asarray(gid_np, dtype=np.int64), minlength=n_groups)
    scores = oracle.edge_scores(Z, w, prefix, lam)
    mag = oracle.edge_scores(np.abs(Z), np.abs(np.asarray(w, dtype=np.float64)), prefix, lam)
    stol = edge_score_tol(scores, mag, Z.shape[2], prefix.shape[1])
    ref_gi, ref_gs = oracle.select(scores, counts, min(k_groups + 1, n_groups))
    if ref_gi.shape[1] == k_groups:
        ref_gi = np.concatenate([ref_gi, -np.ones((len(ref_gi), 1), np.int32)], axis=1)
        ref_gs = np.concatenate([ref_gs, np.full((len(ref_gs), 1), -np.inf)], axis=1)
    ref2 = oracle.stage2(entries_np, gid_np, n_groups, queries_np, gi, k_entries + 16, tau, eps, nthreads)
    qf = _as_f64(queries_np)
    problems = []
    for b in range(queries_np.shape[0]):
        problems += check_ranked(f"query {b} groups", gi[b], gs[b], ref_gi[b], ref_gs[b], k_groups,
                                 lambda g, b=b: float(scores[b, g]), dtype,
                                 tol=lambda g, b=b: float(stol[b, g]))
        problems += _check_entries(ei, es, ew, lse, b, b, ref2, entries_np, qf, k_entries, tau, eps, dtype)
    return problems


def compare_flat(out, entries_np, queries_np, k_entries, tau, eps, dtype, rows=None, nthreads=None):
    """The flat scan of the queries listed in `rows` (all by default) against
    the oracle's flat retrieval."""
    import oracle

    ei = out["entry_idx"].cpu().numpy()
    es = out["entry_score"].cpu().numpy()
    ew = out["entry_weight"].cpu().numpy()
    lse = out["lse"].cpu().numpy()
    rows = np.arange(queries_np.shape[0]) if rows is None else np.asarray(rows)
    q = queries_np[rows]
    ref2 = oracle.flat(entries_np, q, k_entries + 16, tau, eps, nthreads)
    qf = _as_f64(q)
    problems = []
    for r, b in enumerate(rows):
        problems += _check_entries(ei, es, ew, lse, b, r, ref2, entries_np, qf, k_entries, tau, eps, dtype)
    return problems


def check_draws(what, gi, gs, keys, scores, counts, k, dtype, score_tol=None):
    """Groups drawn by the GPU for one query against the oracle's policy keys
    (the index rule on keys: the draws are the top k keys), and their
    group_score against the oracle's float64 scores q . c_g."""
    import oracle

    ref_gi, ref_gk = oracle.select(keys[None, :], counts, min(k + 1, len(counts)))
    ref_gi, ref_gk = ref_gi[0], ref_gk[0]
    if len(ref_gi) == k:
        ref_gi = np.append(ref_gi, -1)
        ref_gk = np.append(ref_gk, -np.inf)
    key_of = [float(keys[g]) if g >= 0 else -np.inf for g in gi]
    problems = check_ranked(what, gi, key_of, ref_gi, ref_gk, k, lambda g: float(keys[g]), dtype)
    for g, s in zip(gi, gs):
        if g < 0:
            continue
        ok = abs(float(s) - scores[g]) <= score_tol[g] if score_tol is not None else close(s, scores[g], dtype)
        if not ok:
            problems.append(f"{what}: score of group {g} gpu {float(s):.7g} oracle {scores[g]:.7g}")
            break
    return problems


def compare_sampled(out, entries_np, gid_np, n_groups, queries_np, k_groups, k_entries, tau, eps, dtype, seed,
                    offset, rows=None, centroid=None, counts=None, scores=None, score_tol=None, nthreads=None):
    """The sampled lookup of the queries in `rows` (all by default): the draws
    against the oracle's policy keys for the same (seed, offset, query),
    stage 2 given the GPU's draws.  `scores` ([B, G] float64) replaces the
    group-key scores (the edge-table router), with `score_tol` ([B, G]) the
    absolute bounds of its values."""
    import oracle

    gi = out["group_idx"].cpu().numpy()
    gs = out["group_score"].cpu().numpy()
    ei = out["entry_idx"].cpu().numpy()
    es = out["entry_score"].cpu().numpy()
    ew = out["entry_weight"].cpu().numpy()
    lse = out["lse"].cpu().numpy()
    B = queries_np.shape[0]
    rows = np.arange(B) if rows is None else np.asarray(rows)
    q = queries_np[rows]
    if counts is None:
        counts = np.bincount(np.asarray(gid_np, dtype=np.int64), minlength=n_groups)
    if scores is None:
        if centroid is None:
            centroid, counts = oracle.centroids(entries_np, gid_np, n_groups, nthreads)
        s_rows = oracle.coarse_scores(q, centroid)
    else:
        s_rows = np.asarray(scores, dtype=np.float64)[rows]
    keys, _ = oracle.policy_keys(s_rows, counts, tau, eps, seed, offset, query_ids=rows)
    ref2 = oracle.stage2(entries_np, gid_np, n_groups, q, gi[rows], k_entries + 16, tau, eps, nthreads)
    qf = _as_f64(q)
    problems = []
    for r, b in enumerate(rows):
        tol_r = None if score_tol is None else np.asarray(score_tol)[b]
        problems += check_draws(f"query {b} draws", gi[b], gs[b], keys[r], s_rows[r], counts, k_groups, dtype,
                                tol_r)
        problems += _check_entries(ei, es, ew, lse, b, r, ref2, entries_np, qf, k_entries, tau, eps, dtype)
    return problems


def _as_f64(x: np.ndarray) -> np.ndarray:
    if x.dtype == np.uint16:
        return (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return x.astype(np.float64)
