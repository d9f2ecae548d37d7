"""Float64 CPU oracle for the hierarchical transition-attended memory lookup.

TEST INFRASTRUCTURE ONLY.  The oracle is the plain definition of what the
lookup computes (group keys, Eq. 9 scoring with the linear scorer of App. B.6,
the Eq. 12 candidate restriction, the Eq. 11 tau-softmax / eps-uniform policy
and the Eq. 13 pick, generalised to top-k).  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it.  It shares no code with the CUDA library and never imports it.

The arithmetic lives in ``htam_oracle.c`` (plain C, double precision,
sequential sums).  This module compiles it with gcc on first use and wraps it
with ctypes; numpy arrays in, numpy arrays out.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "htam_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libhtam_oracle.so")
_lock = threading.Lock()
_lib = None

F32 = 0
BF16 = 1


def build(force: bool = False) -> str:
    """Compile the oracle shared library (gcc, -O2, IEEE semantics kept)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", "-o", tmp, _SRC, "-lpthread", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        lib.htam_oracle_centroid_accumulate.argtypes = [P, ctypes.c_int, P, i64, i32, i32, P, P, ctypes.c_int]
        lib.htam_oracle_centroid_accumulate.restype = ctypes.c_int
        lib.htam_oracle_centroid_finalize.argtypes = [P, P, i32, i32, P]
        lib.htam_oracle_centroid_finalize.restype = None
        lib.htam_oracle_stage1.argtypes = [P, ctypes.c_int, i32, i32, P, P, i32, i32, P, P, ctypes.c_int]
        lib.htam_oracle_stage1.restype = ctypes.c_int
        lib.htam_oracle_stage2.argtypes = [P, ctypes.c_int, P, i64, i32, i32, P, ctypes.c_int, i32, P,
                                           i32, i32, dbl, dbl, P, P, P, P, P, ctypes.c_int]
        lib.htam_oracle_stage2.restype = ctypes.c_int
        lib.htam_oracle_prefix_reduce.argtypes = [P, ctypes.c_int, i32, i32, i32, dbl, P]
        lib.htam_oracle_prefix_reduce.restype = ctypes.c_int
        lib.htam_oracle_edge_scores.argtypes = [P, i32, i32, P, P, i32, i32, dbl, P]
        lib.htam_oracle_edge_scores.restype = ctypes.c_int
        lib.htam_oracle_select.argtypes = [P, P, i32, i32, i32, P, P]
        lib.htam_oracle_select.restype = ctypes.c_int
        lib.htam_oracle_philox4x32_10.argtypes = [P, P, P]
        lib.htam_oracle_philox4x32_10.restype = None
        lib.htam_oracle_policy_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64, i32, i32]
        lib.htam_oracle_policy_uniform.restype = dbl
        lib.htam_oracle_policy_keys.argtypes = [P, P, i32, i32, dbl, dbl, ctypes.c_uint64, ctypes.c_uint64, P, P,
                                                P]
        lib.htam_oracle_policy_keys.restype = ctypes.c_int
        _lib = lib
        return lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _as_input(x: np.ndarray):
    """Return (contiguous array, dtype code). bf16 arrives as uint16 bits."""
    x = np.ascontiguousarray(x)
    if x.dtype == np.float32:
        return x, F32
    if x.dtype == np.uint16:
        return x, BF16
    raise TypeError(f"oracle inputs are float32 or bf16 bits (uint16), got {x.dtype}")


def default_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


class CentroidAccumulator:
    """Group sums and counts fed in chunks (for memories too big to pass at once)."""

    def __init__(self, n_groups: int, d: int):
        self.n_groups, self.d = int(n_groups), int(d)
        self.sums = np.zeros((self.n_groups, self.d), dtype=np.float64)
        self.counts = np.zeros(self.n_groups, dtype=np.int64)

    def add(self, entries: np.ndarray, gid: np.ndarray, nthreads: int | None = None) -> None:
        lib = _load()
        entries, dt = _as_input(entries)
        gid = np.ascontiguousarray(gid, dtype=np.int32)
        n = gid.shape[0]
        if entries.shape != (n, self.d):
            raise ValueError("entries must be [n, d]")
        rc = lib.htam_oracle_centroid_accumulate(_ptr(entries), dt, _ptr(gid), n, self.d,
                                                 self.n_groups, _ptr(self.sums), _ptr(self.counts),
                                                 nthreads or default_threads())
        if rc != 0:
            raise ValueError("group id out of range")

    def finalize(self):
        lib = _load()
        cent = np.empty((self.n_groups, self.d), dtype=np.float64)
        lib.htam_oracle_centroid_finalize(_ptr(self.sums), _ptr(self.counts), self.d,
                                          self.n_groups, _ptr(cent))
        return cent, self.counts.copy()


def centroids(entries: np.ndarray, gid: np.ndarray, n_groups: int, nthreads: int | None = None):
    """Group keys c_g = mean of the group's entries (float64), and counts n_g."""
    acc = CentroidAccumulator(n_groups, entries.shape[1])
    acc.add(entries, gid, nthreads)
    return acc.finalize()


def stage1(queries: np.ndarray, centroid: np.ndarray, counts: np.ndarray, k_groups: int,
           nthreads: int | None = None):
    """Coarse scores against every non-empty group key and the top-k_g groups."""
    lib = _load()
    queries, qdt = _as_input(queries)
    centroid = np.ascontiguousarray(centroid, dtype=np.float64)
    counts = np.ascontiguousarray(counts, dtype=np.int64)
    b, d = queries.shape
    g = centroid.shape[0]
    gi = np.empty((b, k_groups), dtype=np.int32)
    gs = np.empty((b, k_groups), dtype=np.float64)
    rc = lib.htam_oracle_stage1(_ptr(queries), qdt, b, d, _ptr(centroid), _ptr(counts), g,
                                int(k_groups), _ptr(gi), _ptr(gs), nthreads or default_threads())
    if rc != 0:
        raise RuntimeError(f"oracle stage1 failed ({rc})")
    return gi, gs


def stage2(entries: np.ndarray, gid: np.ndarray, n_groups: int, queries: np.ndarray,
           groups: np.ndarray, k_entries: int, tau: float = 1.0, eps: float = 0.0,
           nthreads: int | None = None):
    """Fine scores over the selected groups' entries, softmax and top-k_e.

    ``groups`` is [B, k_g] int32 (-1 = empty slot): the groups each query
    selected.  Returns a dict with entry_idx, entry_score, entry_weight, lse and
    n_cand (the candidate-set size |C_b|).
    """
    lib = _load()
    entries, edt = _as_input(entries)
    queries, qdt = _as_input(queries)
    gid = np.ascontiguousarray(gid, dtype=np.int32)
    groups = np.ascontiguousarray(groups, dtype=np.int32)
    n, d = entries.shape
    b = queries.shape[0]
    kg = groups.shape[1]
    out = {
        "entry_idx": np.empty((b, k_entries), dtype=np.int32),
        "entry_score": np.empty((b, k_entries), dtype=np.float64),
        "entry_weight": np.empty((b, k_entries), dtype=np.float64),
        "lse": np.empty(b, dtype=np.float64),
        "n_cand": np.empty(b, dtype=np.int64),
    }
    rc = lib.htam_oracle_stage2(_ptr(entries), edt, _ptr(gid), n, d, int(n_groups), _ptr(queries),
                                qdt, b, _ptr(groups), kg, int(k_entries), float(tau), float(eps),
                                _ptr(out["entry_idx"]), _ptr(out["entry_score"]),
                                _ptr(out["entry_weight"]), _ptr(out["lse"]), _ptr(out["n_cand"]),
                                nthreads or default_threads())
    if rc != 0:
        raise RuntimeError(f"oracle stage2 failed ({rc})")
    return out


def query(entries: np.ndarray, gid: np.ndarray, n_groups: int, queries: np.ndarray,
          k_groups: int, k_entries: int, tau: float = 1.0, eps: float = 0.0,
          centroid=None, counts=None, nthreads: int | None = None):
    """Full two-level lookup: stage 1 then stage 2 on the groups it selected."""
    if centroid is None or counts is None:
        centroid, counts = centroids(entries, gid, n_groups, nthreads)
    gi, gs = stage1(queries, centroid, counts, k_groups, nthreads)
    out = stage2(entries, gid, n_groups, queries, gi, k_entries, tau, eps, nthreads)
    out["group_idx"] = gi
    out["group_score"] = gs
    return out


def flat(entries: np.ndarray, queries: np.ndarray, k_entries: int, tau: float = 1.0, eps: float = 0.0,
         nthreads: int | None = None):
    """Flat memory retrieval (App. C.4; the "w/o hierarchy" ablation of
    App. C.8): every entry is a candidate and there is no group stage.  Stage 2
    over a memory of one group that holds all n entries: fine scores against
    all of them, the softmax of Eq. 11 with |C| = n, the top-k_e of Eq. 13."""
    n = entries.shape[0]
    b = queries.shape[0]
    return stage2(entries, np.zeros(n, np.int32), 1, queries, np.zeros((b, 1), np.int32), k_entries, tau, eps,
                  nthreads)


def prefix_reduce(prefix: np.ndarray, lam: float) -> np.ndarray:
    """Prefix-attended query (Eq. 9 over the prefix of Eq. 8, weights of
    Eq. 10): prefix [b, P, d] (q_P the most recent) -> qbar [b, d] float64,
    qbar = sum_i exp(-lam * (P - i)) * q_i.  By linearity of the scorer,
    qbar . c_g is the prefix score of group g."""
    lib = _load()
    prefix, dt = _as_input(prefix)
    b, p_len, d = prefix.shape
    out = np.empty((b, d), dtype=np.float64)
    rc = lib.htam_oracle_prefix_reduce(_ptr(prefix), dt, b, p_len, d, float(lam), _ptr(out))
    if rc != 0:
        raise ValueError("oracle prefix_reduce: bad argument")
    return out


def round_query(x: np.ndarray, dtype: str) -> np.ndarray:
    """A float64 query rounded to the memory's dtype as the lookup consumes
    it: float32 (round to nearest even), or bf16 bits via float32 (each step
    round to nearest even)."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    if dtype == "f32":
        return f
    u = f.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def edge_scores(Z: np.ndarray, w: np.ndarray, prefix: np.ndarray, lam: float) -> np.ndarray:
    """Edge-table router scores (Eq. 9 with the App. B.6 utility phi = w . z
    and the Eq. 10 weights): Z [G, G, F] float32 (from, to, feature), w [F],
    prefix [b, P] int32 group ids (-1 = none) -> [b, G] float64."""
    lib = _load()
    Z = np.ascontiguousarray(Z, dtype=np.float32)
    G, G2, F = Z.shape
    if G2 != G:
        raise ValueError("Z must be [G, G, F]")
    w = np.ascontiguousarray(w, dtype=np.float64)
    prefix = np.ascontiguousarray(prefix, dtype=np.int32)
    b, p_len = prefix.shape
    out = np.empty((b, G), dtype=np.float64)
    rc = lib.htam_oracle_edge_scores(_ptr(Z), G, F, _ptr(w), _ptr(prefix), b, p_len, float(lam), _ptr(out))
    if rc != 0:
        raise ValueError("oracle edge_scores: bad argument")
    return out


def select(scores: np.ndarray, counts: np.ndarray, k: int):
    """The k best groups of per-group scores, ranked like stage 1 (score
    descending, ties to the lower id, empty groups excluded, -1/-inf padding)."""
    lib = _load()
    scores = np.ascontiguousarray(scores, dtype=np.float64)
    counts = np.ascontiguousarray(counts, dtype=np.int64)
    b, G = scores.shape
    gi = np.empty((b, k), dtype=np.int32)
    gs = np.empty((b, k), dtype=np.float64)
    if lib.htam_oracle_select(_ptr(scores), _ptr(counts), b, G, int(k), _ptr(gi), _ptr(gs)) != 0:
        raise MemoryError("oracle select")
    return gi, gs


def query_edges(entries: np.ndarray, gid: np.ndarray, n_groups: int, Z: np.ndarray, w: np.ndarray,
                prefix: np.ndarray, lam: float, queries: np.ndarray, k_groups: int, k_entries: int,
                tau: float = 1.0, eps: float = 0.0, nthreads: int | None = None):
    """The lookup with the edge-table router as stage 1 (the paper's global
    direction choice) and the query embeddings for stage 2 (the local pick)."""
    counts = np.bincount(np.asarray(gid, dtype=np.int64), minlength=n_groups)
    gi, gs = select(edge_scores(Z, w, prefix, lam), counts, k_groups)
    out = stage2(entries, gid, n_groups, queries, gi, k_entries, tau, eps, nthreads)
    out["group_idx"] = gi
    out["group_score"] = gs
    return out


def assign_nearest(entries: np.ndarray, gid: np.ndarray, centroid: np.ndarray, counts: np.ndarray,
                   nthreads: int | None = None) -> np.ndarray:
    """Group ids of appended entries: ids >= 0 kept, each -1 replaced by the
    group whose key scores highest against the entry (stage 1's scorer and
    ranking with k_g = 1: ties to the lower id, empty groups excluded), with
    the keys as they stand before the append."""
    out = np.array(gid, dtype=np.int32, copy=True)
    miss = np.flatnonzero(out == -1)
    if len(miss):
        gi, _ = stage1(np.ascontiguousarray(np.asarray(entries)[miss]), centroid, counts, 1, nthreads)
        out[miss] = gi[:, 0]
    return out


# ------------------------------------------------ sampling from the policy (Eq. 11)

def philox4x32_10(ctr, key) -> np.ndarray:
    """Philox4x32-10 (Salmon et al., SC 2011): four counter words and two key
    words (uint32) -> four uint32 outputs."""
    lib = _load()
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    if c.shape != (4,) or k.shape != (2,):
        raise ValueError("counter has 4 words, key 2")
    out = np.empty(4, dtype=np.uint32)
    lib.htam_oracle_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def policy_uniform(seed: int, offset: int, b: int, g: int) -> float:
    """The uniform in (0, 1) that query b draws for group g."""
    return float(_load().htam_oracle_policy_uniform(seed, offset, b, g))


def coarse_scores(queries: np.ndarray, centroid: np.ndarray) -> np.ndarray:
    """s[b][g] = q_b . c_g in float64 for every group (matrix product)."""
    return _as_f64_input(queries) @ np.asarray(centroid, dtype=np.float64).T


def policy_keys(scores: np.ndarray, counts: np.ndarray, tau: float, eps: float, seed: int, offset: int,
                query_ids=None):
    """Gumbel-top-k keys of the Eq. 11 policy over the non-empty groups and
    the policy itself: returns (keys, mu), both [b, G] float64.  Row r draws
    with the uniforms of query query_ids[r] (default r)."""
    lib = _load()
    scores = np.ascontiguousarray(scores, dtype=np.float64)
    counts = np.ascontiguousarray(counts, dtype=np.int64)
    b, G = scores.shape
    ids = None if query_ids is None else np.ascontiguousarray(query_ids, dtype=np.int32)
    if ids is not None and ids.shape != (b,):
        raise ValueError("query_ids must have one id per row")
    keys = np.empty((b, G), dtype=np.float64)
    mu = np.empty((b, G), dtype=np.float64)
    rc = lib.htam_oracle_policy_keys(_ptr(scores), _ptr(counts), b, G, float(tau), float(eps), int(seed),
                                     int(offset), _ptr(ids) if ids is not None else None, _ptr(keys), _ptr(mu))
    if rc != 0:
        raise ValueError("oracle policy_keys: bad argument")
    return keys, mu


def query_sampled(entries: np.ndarray, gid: np.ndarray, n_groups: int, queries: np.ndarray, k_groups: int,
                  k_entries: int, tau: float, eps: float, seed: int, offset: int, centroid=None, counts=None,
                  nthreads: int | None = None):
    """The lookup with stage 1 drawn from the policy (Algorithm 1, step 2:
    k_groups draws without replacement from mu_g of Eq. 11 over the group-key
    scores), then stage 2 on the drawn groups."""
    if centroid is None or counts is None:
        centroid, counts = centroids(entries, gid, n_groups, nthreads)
    keys, mu = policy_keys(coarse_scores(queries, centroid), counts, tau, eps, seed, offset)
    gi, gk = select(keys, counts, k_groups)
    out = stage2(entries, gid, n_groups, queries, gi, k_entries, tau, eps, nthreads)
    out["group_idx"] = gi
    out["group_key"] = gk
    out["keys"] = keys
    out["mu"] = mu
    return out


def _as_f64_input(x: np.ndarray) -> np.ndarray:
    """float32 arrays or bf16 bit patterns (uint16) as float64, exactly."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        return (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return x.astype(np.float64)
