"""Python binding of the C ABI in include/htam.h (argument marshalling only).

Every step of the lookup runs in the CUDA library ``_lib/libhtam.so``; this
module passes torch tensors' device pointers and the current CUDA stream
through ctypes.  There is no fallback: if the library is missing the import
fails, and every call raises on a non-OK status.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libhtam.so")

HTAM_OK, HTAM_EINVAL, HTAM_ENOMEM, HTAM_ECAPACITY, HTAM_ECUDA, HTAM_ETIMEOUT, HTAM_ENODEV = range(7)
HTAM_F32, HTAM_BF16 = 0, 1
HTAM_TUNE_TC_MIN_BUCKET, HTAM_TUNE_STREAM_ROWS, HTAM_TUNE_TC_PAIRS, HTAM_TUNE_PDL = 0, 1, 2, 3
HTAM_TUNE_FINE_OVERLAP = 4
HTAM_MAX_PREFIX = 64  # longest prefix htam_query_prefix takes
HTAM_MAX_EDGE_FEATURES = 32  # most features per edge htam_query_edges takes

# Every symbol include/htam.h declares, in declaration order.
EXPORTS = (
    "htam_build_memory", "htam_append_transitions", "htam_append_assign", "htam_query", "htam_query_host",
    "htam_query_prefix", "htam_query_edges", "htam_query_sampled", "htam_query_edges_sampled", "htam_query_flat",
    "htam_select_groups_static", "htam_memory_info", "htam_memory_group_counts", "htam_memory_group_keys",
    "htam_device_status", "htam_set_tuning", "htam_get_tuning", "htam_set_phase_timing",
    "htam_read_phase_timing", "htam_free_memory", "htam_status_string", "htam_last_error",
    "htam_selftest_wait_timeout",
)
PHASES = ("coarse", "select", "bucket", "fine", "fine_tc", "merge", "prefix", "append")


class HtamError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        msg = _lib.htam_status_string(status).decode()
        detail = _lib.htam_last_error().decode()
        super().__init__(f"{what}: {msg}" + (f" ({detail})" if detail and status == HTAM_ECUDA else ""))


class QueryParams(ctypes.Structure):
    _fields_ = [("k_groups", ctypes.c_int32), ("k_entries", ctypes.c_int32),
                ("tau", ctypes.c_float), ("epsilon", ctypes.c_float)]


class Sampling(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("offset", ctypes.c_uint64)]


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2605_29734_gb300.build.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, i32, i64, st = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int
    PP = ctypes.POINTER(ctypes.c_void_p)
    lib.htam_build_memory.argtypes = [P, P, i64, i32, i32, ctypes.c_int, i64, P, PP]
    lib.htam_append_transitions.argtypes = [P, P, P, i64, P]
    lib.htam_append_assign.argtypes = [P, P, P, i64, P, P]
    qargs = [P, P, i32, ctypes.POINTER(QueryParams), P, P, P, P, P, P, P]
    lib.htam_query.argtypes = qargs
    lib.htam_query_host.argtypes = qargs
    lib.htam_query_prefix.argtypes = [P, P, i32, i32, ctypes.c_float, ctypes.POINTER(QueryParams),
                                      P, P, P, P, P, P, P]
    lib.htam_query_edges.argtypes = [P, P, i32, P, P, i32, ctypes.c_float, P, i32, ctypes.POINTER(QueryParams),
                                     P, P, P, P, P, P, P]
    lib.htam_query_sampled.argtypes = [P, P, i32, ctypes.POINTER(QueryParams), ctypes.POINTER(Sampling),
                                       P, P, P, P, P, P, P]
    lib.htam_query_edges_sampled.argtypes = [P, P, i32, P, P, i32, ctypes.c_float, P, i32,
                                             ctypes.POINTER(QueryParams), ctypes.POINTER(Sampling),
                                             P, P, P, P, P, P, P]
    lib.htam_query_flat.argtypes = [P, P, i32, i32, ctypes.c_float, ctypes.c_float, P, P, P, P, P]
    lib.htam_memory_info.argtypes = [P, P, P, P, P]
    lib.htam_memory_group_counts.argtypes = [P, P]
    lib.htam_memory_group_keys.argtypes = [P, P, P]
    lib.htam_device_status.argtypes = [P, P]
    lib.htam_free_memory.argtypes = [P]
    lib.htam_free_memory.restype = None
    lib.htam_status_string.argtypes = [st]
    lib.htam_status_string.restype = ctypes.c_char_p
    lib.htam_last_error.argtypes = []
    lib.htam_last_error.restype = ctypes.c_char_p
    lib.htam_selftest_wait_timeout.argtypes = [i64, P]
    lib.htam_select_groups_static.argtypes = [P, P, i32, i32, P, P, P]
    lib.htam_select_groups_static.restype = st
    lib.htam_set_tuning.argtypes = [P, ctypes.c_int, i32]
    lib.htam_set_tuning.restype = st
    lib.htam_get_tuning.argtypes = [P, ctypes.c_int, ctypes.POINTER(i32)]
    lib.htam_get_tuning.restype = st
    lib.htam_set_phase_timing.argtypes = [P, ctypes.c_int]
    lib.htam_read_phase_timing.argtypes = [P, P, P, P, P]
    for name in ("htam_build_memory", "htam_append_transitions", "htam_query", "htam_query_host",
                 "htam_memory_info", "htam_memory_group_counts", "htam_memory_group_keys",
                 "htam_device_status", "htam_selftest_wait_timeout", "htam_set_phase_timing",
                 "htam_read_phase_timing"):
        getattr(lib, name).restype = st
    return lib


_lib = _load()


def lib() -> ctypes.CDLL:
    return _lib


def _check(status: int, what: str) -> None:
    if status != HTAM_OK:
        raise HtamError(status, what)


def _stream_ptr(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(stream.cuda_stream))


def _dev_ptr(t: torch.Tensor | None) -> ctypes.c_void_p:
    if t is None:
        return ctypes.c_void_p(0)
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CUDA tensor")
    return ctypes.c_void_p(t.data_ptr())


def _dtype_code(dt: torch.dtype) -> int:
    if dt == torch.bfloat16:
        return HTAM_BF16
    if dt == torch.float32:
        return HTAM_F32
    raise TypeError(f"entries must be bfloat16 or float32, got {dt}")


class Memory:
    """A device-resident two-level memory (groups of transition entries)."""

    def __init__(self, entries: torch.Tensor, group_ids: torch.Tensor, n_groups: int,
                 capacity: int | None = None, stream=None):
        if entries.dim() != 2 or group_ids.dim() != 1 or group_ids.dtype != torch.int32:
            raise ValueError("entries [n, d] and int32 group_ids [n] expected")
        n, d = entries.shape
        self.dtype = entries.dtype
        self.d = int(d)
        self.n_groups = int(n_groups)
        handle = ctypes.c_void_p()
        cap = int(capacity if capacity is not None else max(n, 1))
        _check(_lib.htam_build_memory(_dev_ptr(entries), _dev_ptr(group_ids), n, d, n_groups,
                                      _dtype_code(entries.dtype), cap, _stream_ptr(stream),
                                      ctypes.byref(handle)), "htam_build_memory")
        self._h = handle

    @property
    def handle(self) -> ctypes.c_void_p:
        if not self._h:
            raise RuntimeError("memory already freed")
        return self._h

    def append(self, entries: torch.Tensor, group_ids: torch.Tensor, stream=None, check: bool = False) -> None:
        """Queues an append (no host round trip).  Group ids are checked on
        the device: a rejected batch changes nothing and is reported by
        device_status(); check=True waits for that report and raises it."""
        if entries.dtype != self.dtype or group_ids.dtype != torch.int32:
            raise TypeError("entries must match the memory dtype; group_ids int32")
        if entries.dim() != 2 or entries.shape[1] != self.d or group_ids.shape[0] != entries.shape[0]:
            raise ValueError("entries [count, d] and group_ids [count] expected")
        _check(_lib.htam_append_transitions(self.handle, _dev_ptr(entries), _dev_ptr(group_ids),
                                            entries.shape[0], _stream_ptr(stream)),
               "htam_append_transitions")
        if check:
            _check(self.device_status(stream), "htam_append_transitions (device check)")

    def append_assign(self, entries: torch.Tensor, group_ids: torch.Tensor, stream=None,
                      check: bool = False) -> torch.Tensor:
        """append() that returns the group each entry joined (ids of -1 join
        the group with the nearest key)."""
        if entries.dtype != self.dtype or group_ids.dtype != torch.int32:
            raise TypeError("entries must match the memory dtype; group_ids int32")
        if entries.dim() != 2 or entries.shape[1] != self.d or group_ids.shape[0] != entries.shape[0]:
            raise ValueError("entries [count, d] and group_ids [count] expected")
        assigned = torch.empty_like(group_ids)
        _check(_lib.htam_append_assign(self.handle, _dev_ptr(entries), _dev_ptr(group_ids), entries.shape[0],
                                       _dev_ptr(assigned), _stream_ptr(stream)), "htam_append_assign")
        if check:
            _check(self.device_status(stream), "htam_append_assign (device check)")
        return assigned

    def query(self, queries: torch.Tensor, k_groups: int, k_entries: int, tau: float = 1.0,
              epsilon: float = 0.0, stream=None, out: dict | None = None) -> dict:
        """Device lookup; returns (or fills) a dict of device tensors."""
        b, out = self._lookup_out(queries, k_groups, k_entries, out)
        p = QueryParams(k_groups, k_entries, tau, epsilon)
        _check(_lib.htam_query(self.handle, _dev_ptr(queries), b, ctypes.byref(p),
                               _dev_ptr(out["group_idx"]), _dev_ptr(out["group_score"]),
                               _dev_ptr(out["entry_idx"]), _dev_ptr(out["entry_score"]),
                               _dev_ptr(out["entry_weight"]), _dev_ptr(out.get("lse")),
                               _stream_ptr(stream)), "htam_query")
        return out

    def query_sampled(self, queries: torch.Tensor, k_groups: int, k_entries: int, seed: int, offset: int,
                      tau: float = 1.0, epsilon: float = 0.0, stream=None, out: dict | None = None) -> dict:
        """Lookup with the groups drawn from the policy of Eq. 11 (k_groups
        draws without replacement; Philox uniforms from seed and offset)."""
        b, out = self._lookup_out(queries, k_groups, k_entries, out)
        p = QueryParams(k_groups, k_entries, tau, epsilon)
        smp = Sampling(seed, offset)
        _check(_lib.htam_query_sampled(self.handle, _dev_ptr(queries), b, ctypes.byref(p), ctypes.byref(smp),
                                       _dev_ptr(out["group_idx"]), _dev_ptr(out["group_score"]),
                                       _dev_ptr(out["entry_idx"]), _dev_ptr(out["entry_score"]),
                                       _dev_ptr(out["entry_weight"]), _dev_ptr(out.get("lse")),
                                       _stream_ptr(stream)), "htam_query_sampled")
        return out

    def _lookup_out(self, queries: torch.Tensor, k_groups: int, k_entries: int, out: dict | None):
        if queries.dtype != self.dtype or queries.dim() != 2 or queries.shape[1] != self.d:
            raise ValueError("queries must be [b, d] of the memory dtype")
        b = queries.shape[0]
        dev = queries.device
        if out is None:
            out = {
                "group_idx": torch.empty(b, k_groups, dtype=torch.int32, device=dev),
                "group_score": torch.empty(b, k_groups, dtype=torch.float32, device=dev),
                "entry_idx": torch.empty(b, k_entries, dtype=torch.int32, device=dev),
                "entry_score": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "entry_weight": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "lse": torch.empty(b, dtype=torch.float32, device=dev),
            }
        return b, out

    def query_flat(self, queries: torch.Tensor, k_entries: int, tau: float = 1.0, epsilon: float = 0.0,
                   stream=None, out: dict | None = None) -> dict:
        """Flat scan: every entry a candidate, no group stage; returns (or
        fills) entry_idx, entry_score, entry_weight and lse."""
        if queries.dtype != self.dtype or queries.dim() != 2 or queries.shape[1] != self.d:
            raise ValueError("queries must be [b, d] of the memory dtype")
        b = queries.shape[0]
        dev = queries.device
        if out is None:
            out = {
                "entry_idx": torch.empty(b, k_entries, dtype=torch.int32, device=dev),
                "entry_score": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "entry_weight": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "lse": torch.empty(b, dtype=torch.float32, device=dev),
            }
        _check(_lib.htam_query_flat(self.handle, _dev_ptr(queries), b, k_entries, float(tau), float(epsilon),
                                    _dev_ptr(out["entry_idx"]), _dev_ptr(out["entry_score"]),
                                    _dev_ptr(out["entry_weight"]), _dev_ptr(out.get("lse")),
                                    _stream_ptr(stream)), "htam_query_flat")
        return out

    def query_prefix(self, prefix: torch.Tensor, lam: float, k_groups: int, k_entries: int, tau: float = 1.0,
                     epsilon: float = 0.0, stream=None, out: dict | None = None) -> dict:
        """Prefix-attended lookup: prefix [b, P, d] of the memory dtype (the
        most recent state last), position weights exp(-lam * (P - i))."""
        if prefix.dtype != self.dtype or prefix.dim() != 3 or prefix.shape[2] != self.d:
            raise ValueError("prefix must be [b, P, d] of the memory dtype")
        b, p_len = prefix.shape[0], prefix.shape[1]
        dev = prefix.device
        if out is None:
            out = {
                "group_idx": torch.empty(b, k_groups, dtype=torch.int32, device=dev),
                "group_score": torch.empty(b, k_groups, dtype=torch.float32, device=dev),
                "entry_idx": torch.empty(b, k_entries, dtype=torch.int32, device=dev),
                "entry_score": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "entry_weight": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "lse": torch.empty(b, dtype=torch.float32, device=dev),
            }
        p = QueryParams(k_groups, k_entries, tau, epsilon)
        _check(_lib.htam_query_prefix(self.handle, _dev_ptr(prefix), b, p_len, float(lam), ctypes.byref(p),
                                      _dev_ptr(out["group_idx"]), _dev_ptr(out["group_score"]),
                                      _dev_ptr(out["entry_idx"]), _dev_ptr(out["entry_score"]),
                                      _dev_ptr(out["entry_weight"]), _dev_ptr(out.get("lse")),
                                      _stream_ptr(stream)), "htam_query_prefix")
        return out

    def query_edges(self, edge_features: torch.Tensor, weights, prefix_groups, lam: float, queries: torch.Tensor,
                    k_groups: int, k_entries: int, tau: float = 1.0, epsilon: float = 0.0, stream=None,
                    out: dict | None = None, sampling: tuple[int, int] | None = None) -> dict:
        """Lookup routed by transition edges: edge_features [G, G, F] float32
        on the device, weights [F] and prefix_groups [b, P] (int32, -1 = none)
        on the host, queries [b, d] on the device for the entry level.  With
        sampling = (seed, offset) the groups are drawn from the policy of
        Eq. 11 over the edge scores instead of ranked."""
        if edge_features.dtype != torch.float32 or edge_features.dim() != 3:
            raise ValueError("edge_features must be a [G, G, F] float32 tensor")
        if queries.dtype != self.dtype or queries.dim() != 2 or queries.shape[1] != self.d:
            raise ValueError("queries must be [b, d] of the memory dtype")
        w = torch.as_tensor(weights, dtype=torch.float32).contiguous().cpu()
        pre = torch.as_tensor(prefix_groups, dtype=torch.int32).contiguous().cpu()
        b = queries.shape[0]
        if pre.dim() != 2 or pre.shape[0] != b:
            raise ValueError("prefix_groups must be [b, P]")
        dev = queries.device
        if out is None:
            out = {
                "group_idx": torch.empty(b, k_groups, dtype=torch.int32, device=dev),
                "group_score": torch.empty(b, k_groups, dtype=torch.float32, device=dev),
                "entry_idx": torch.empty(b, k_entries, dtype=torch.int32, device=dev),
                "entry_score": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "entry_weight": torch.empty(b, k_entries, dtype=torch.float32, device=dev),
                "lse": torch.empty(b, dtype=torch.float32, device=dev),
            }
        p = QueryParams(k_groups, k_entries, tau, epsilon)
        head = (self.handle, _dev_ptr(edge_features), edge_features.shape[2], ctypes.c_void_p(w.data_ptr()),
                ctypes.c_void_p(pre.data_ptr()), pre.shape[1], float(lam), _dev_ptr(queries), b, ctypes.byref(p))
        tail = (_dev_ptr(out["group_idx"]), _dev_ptr(out["group_score"]), _dev_ptr(out["entry_idx"]),
                _dev_ptr(out["entry_score"]), _dev_ptr(out["entry_weight"]), _dev_ptr(out.get("lse")),
                _stream_ptr(stream))
        if sampling is None:
            _check(_lib.htam_query_edges(*head, *tail), "htam_query_edges")
        else:
            smp = Sampling(*sampling)
            _check(_lib.htam_query_edges_sampled(*head, ctypes.byref(smp), *tail), "htam_query_edges_sampled")
        return out

    def query_host(self, queries: torch.Tensor, k_groups: int, k_entries: int, tau: float = 1.0,
                   epsilon: float = 0.0, stream=None, out: dict | None = None) -> dict:
        """Lookup with host (CPU, ideally pinned) tensors in and out; the copies
        to and from the device happen inside the library call."""
        if queries.is_cuda or not queries.is_contiguous():
            raise ValueError("query_host takes a contiguous CPU tensor")
        b = queries.shape[0]
        pin = queries.is_pinned()
        if out is None:
            def mk(shape, dt):
                return torch.empty(shape, dtype=dt, pin_memory=pin)
            out = {"group_idx": mk((b, k_groups), torch.int32), "group_score": mk((b, k_groups), torch.float32),
                   "entry_idx": mk((b, k_entries), torch.int32), "entry_score": mk((b, k_entries), torch.float32),
                   "entry_weight": mk((b, k_entries), torch.float32), "lse": mk((b,), torch.float32)}
        p = QueryParams(k_groups, k_entries, tau, epsilon)
        hp = lambda t: ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)
        _check(_lib.htam_query_host(self.handle, hp(queries), b, ctypes.byref(p), hp(out["group_idx"]),
                                    hp(out["group_score"]), hp(out["entry_idx"]), hp(out["entry_score"]),
                                    hp(out["entry_weight"]), hp(out.get("lse")), _stream_ptr(stream)),
               "htam_query_host")
        return out

    def info(self) -> dict:
        n, d, g, cap = ctypes.c_int64(), ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int64()
        _check(_lib.htam_memory_info(self.handle, ctypes.byref(n), ctypes.byref(d), ctypes.byref(g),
                                     ctypes.byref(cap)), "htam_memory_info")
        return {"n": n.value, "d": d.value, "n_groups": g.value, "capacity": cap.value}

    def group_counts(self) -> torch.Tensor:
        out = torch.empty(self.n_groups, dtype=torch.int64)
        _check(_lib.htam_memory_group_counts(self.handle, ctypes.c_void_p(out.data_ptr())),
               "htam_memory_group_counts")
        return out

    def group_keys(self, stream=None) -> torch.Tensor:
        out = torch.empty(self.n_groups, self.d, dtype=torch.float32)
        _check(_lib.htam_memory_group_keys(self.handle, ctypes.c_void_p(out.data_ptr()), _stream_ptr(stream)),
               "htam_memory_group_keys")
        return out

    def device_status(self, stream=None) -> int:
        return _lib.htam_device_status(self.handle, _stream_ptr(stream))

    def set_tuning(self, key: int, value: int) -> None:
        _check(_lib.htam_set_tuning(self.handle, int(key), int(value)), "htam_set_tuning")

    def get_tuning(self, key: int) -> int:
        v = ctypes.c_int32()
        _check(_lib.htam_get_tuning(self.handle, int(key), ctypes.byref(v)), "htam_get_tuning")
        return v.value

    def set_tensor_core_min_bucket(self, min_bucket: int) -> None:
        """Buckets of at least `min_bucket` queries go to the tensor-core kernel."""
        self.set_tuning(HTAM_TUNE_TC_MIN_BUCKET, min_bucket)

    def set_stream_rows(self, enable: bool) -> None:
        """CUDA-core path: stream rows through shared memory (True) or load
        them directly (False)."""
        self.set_tuning(HTAM_TUNE_STREAM_ROWS, int(bool(enable)))

    def set_tensor_core_pairs(self, enable: bool) -> None:
        """Tensor-core buckets of more than 128 queries on SM pairs (True) or
        single SMs (False)."""
        self.set_tuning(HTAM_TUNE_TC_PAIRS, int(bool(enable)))

    def set_fine_overlap(self, enable: bool) -> None:
        """CUDA-core and tensor-core fine kernels concurrently (True, default)
        or one after the other (False)."""
        self.set_tuning(HTAM_TUNE_FINE_OVERLAP, int(bool(enable)))

    def set_programmatic_launch(self, enable: bool) -> None:
        """Kernels of a query or append launched with programmatic stream
        serialisation (True, default) or plainly (False)."""
        self.set_tuning(HTAM_TUNE_PDL, int(bool(enable)))

    def set_phase_timing(self, enable: bool) -> None:
        _check(_lib.htam_set_phase_timing(self.handle, int(bool(enable))), "htam_set_phase_timing")

    def read_phase_timing(self, stream=None) -> dict:
        """{phase: (device ms summed, kernel launches)} plus 'queries', since the last read."""
        n = len(PHASES)
        ms = (ctypes.c_double * n)()
        launches = (ctypes.c_int64 * n)()
        queries = ctypes.c_int64()
        _check(_lib.htam_read_phase_timing(self.handle, ms, launches, ctypes.byref(queries), _stream_ptr(stream)),
               "htam_read_phase_timing")
        out = {p: (ms[i], launches[i]) for i, p in enumerate(PHASES)}
        out["queries"] = queries.value
        return out

    def close(self) -> None:
        if self._h:
            _lib.htam_free_memory(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):  # pragma: no cover - best effort
        try:
            self.close()
        except Exception:
            pass


def selftest_wait_timeout(max_iters: int, stream=None) -> int:
    """Runs the bounded-wait diagnostic; returns the status code."""
    return _lib.htam_selftest_wait_timeout(int(max_iters), _stream_ptr(stream))
