"""Seeded synthetic workloads for the memory lookup.

This module only makes inputs: group sizes, group ids, entry and query
embeddings, append batches.  It holds none of the lookup's arithmetic, and both
the CUDA path and the float64 oracle consume the arrays it returns.

Recipe (the paper measures no lookup workload of its own; these shapes stand
in for a memory of global/local nodes at scale):
  * group sizes: ``uniform_random`` (each entry's group drawn uniformly),
    ``uniform`` (n/G entries per group) or ``zipf`` (n_r proportional to
    r^-1.1 for rank r = 1..G, largest-remainder rounding to sum n, at least 1
    per group; group id = r - 1);
  * the entry order is shuffled, so a build must sort by group;
  * ``gaussian`` embeddings: N(0, 1) per coordinate, then L2-normalised;
  * ``clustered`` embeddings: a group centre drawn N(0, 1) per coordinate,
    plus N(0, 0.3^2) noise (0.3 is the standard deviation), L2-normalised;
  * queries: ``gaussian`` ones are N(0, 1) normalised; ``clustered`` ones take
    the centre of the group of a uniformly drawn entry (so a group is chosen
    in proportion to its size), add N(0, 0.3^2) noise and normalise;
  * values are made in float32; bf16 workloads round the normalised float32
    values to bf16 with round-to-nearest-even, and both sides read the same
    bf16 arrays.
Generation uses torch generators on the requested device; the same seed gives
different numbers on CPU and CUDA, so a test generates once and hands the
same arrays to both sides.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    b: int            # queries per batch
    d: int            # embedding dimension
    dtype: str        # "f32" or "bf16"
    g: int            # groups
    n: int            # entries in the memory (initial entries for streaming)
    sizes: str        # "uniform_random" | "uniform" | "zipf"
    embed: str        # "gaussian" | "clustered"
    k_groups: int
    k_entries: int
    rounds: int = 0           # streaming: append+query rounds
    append_per_round: int = 0
    noise: float = 0.3
    zipf_s: float = 1.1

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def capacity(self) -> int:
        return self.n + self.rounds * self.append_per_round


WORKLOADS = {
    # 8 queries, dim 256 fp32, 16 groups, 1,024 entries, top-4 groups / top-4 entries
    "tiny_f32_1k": Workload("tiny_f32_1k", 8, 256, "f32", 16, 1024, "uniform_random",
                            "gaussian", 4, 4),
    # 256 queries, dim 1024 bf16, 256 groups, 65,536 Zipf(1.1) entries, top-8 / top-16
    "zipf_bf16_65k": Workload("zipf_bf16_65k", 256, 1024, "bf16", 256, 65536, "zipf",
                              "clustered", 8, 16),
    # 4,096 queries, dim 1024 bf16, 1,024 groups, 1,048,576 Zipf entries, top-16 / top-32
    "zipf_bf16_1m": Workload("zipf_bf16_1m", 4096, 1024, "bf16", 1024, 1048576, "zipf",
                             "clustered", 16, 32),
    # 64 queries, dim 4096 bf16, 4,096 groups x 1,024 entries (32 GiB of keys), top-32 / top-16
    "uniform_bf16_4m": Workload("uniform_bf16_4m", 64, 4096, "bf16", 4096, 4194304, "uniform",
                                "clustered", 32, 16),
    # 524,288 entries dim 1024 bf16, 512 Zipf groups; 100 rounds of
    # (append 4,096 entries, then 1,024 queries), top-8 / top-16
    "stream_bf16_512k": Workload("stream_bf16_512k", 1024, 1024, "bf16", 512, 524288, "zipf",
                                 "clustered", 8, 16, rounds=100, append_per_round=4096),
}


def zipf_sizes(n: int, g: int, s: float = 1.1) -> np.ndarray:
    """Deterministic Zipf(s) group sizes summing to n, each at least 1."""
    if n < g:
        raise ValueError("zipf sizes need n >= g")
    w = np.arange(1, g + 1, dtype=np.float64) ** (-s)
    extra = n - g                      # one entry per group first
    share = w / w.sum() * extra
    base = np.floor(share).astype(np.int64)
    rem = extra - int(base.sum())
    order = np.argsort(-(share - base), kind="stable")
    base[order[:rem]] += 1
    return base + 1


def _gen(seed: int, stream: int, device) -> torch.Generator:
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) * 1_000_003 + int(stream))
    return gen


def group_sizes(w: Workload) -> np.ndarray | None:
    if w.sizes == "zipf":
        return zipf_sizes(w.n, w.g, w.zipf_s)
    if w.sizes == "uniform":
        if w.n % w.g:
            raise ValueError("uniform sizes need n divisible by g")
        return np.full(w.g, w.n // w.g, dtype=np.int64)
    return None


def make_group_ids(w: Workload, seed: int = 0, device="cpu") -> torch.Tensor:
    """[n] int32 group ids in shuffled (ungrouped) order."""
    gen = _gen(seed, 1, device)
    if w.sizes == "uniform_random":
        return torch.randint(0, w.g, (w.n,), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
    sizes = torch.as_tensor(group_sizes(w), device=device)
    gid = torch.repeat_interleave(torch.arange(w.g, device=device), sizes)
    perm = torch.randperm(w.n, generator=gen, device=device)
    return gid[perm].to(torch.int32).contiguous()


def make_centres(w: Workload, seed: int = 0, device="cpu") -> torch.Tensor:
    return torch.randn(w.g, w.d, generator=_gen(seed, 2, device), device=device, dtype=torch.float32)


def _finish(x: torch.Tensor, dtype) -> torch.Tensor:
    x = x / torch.linalg.vector_norm(x, dim=1, keepdim=True)
    return x.to(dtype)


def make_rows(w: Workload, gid: torch.Tensor, centres: torch.Tensor | None, gen: torch.Generator,
              out: torch.Tensor | None = None, chunk: int = 1 << 18) -> torch.Tensor:
    """Embeddings for the given group ids ([len(gid), d] of the workload dtype)."""
    device = gid.device
    n = gid.shape[0]
    if out is None:
        out = torch.empty(n, w.d, dtype=w.torch_dtype, device=device)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        noise = torch.randn(e - s, w.d, generator=gen, device=device, dtype=torch.float32)
        if w.embed == "clustered":
            x = centres[gid[s:e].long()] + w.noise * noise
        else:
            x = noise
        out[s:e] = _finish(x, w.torch_dtype)
    return out


def make_memory(w: Workload, seed: int = 0, device="cpu"):
    """Returns (entries [n, d], group_ids [n] int32, centres [g, d] float32 or None)."""
    gid = make_group_ids(w, seed, device)
    centres = make_centres(w, seed, device) if w.embed == "clustered" else None
    entries = make_rows(w, gid, centres, _gen(seed, 3, device))
    return entries, gid, centres


def make_queries(w: Workload, gid: torch.Tensor, centres: torch.Tensor | None, seed: int = 0,
                 b: int | None = None, stream: int = 4) -> torch.Tensor:
    """[b, d] queries of the workload dtype (see the module recipe)."""
    device = gid.device
    b = w.b if b is None else b
    gen = _gen(seed, stream, device)
    if w.embed == "clustered":
        pick = torch.randint(0, gid.shape[0], (b,), generator=gen, device=device)
        home = gid[pick]
        noise = torch.randn(b, w.d, generator=gen, device=device, dtype=torch.float32)
        x = centres[home.long()] + w.noise * noise
    else:
        x = torch.randn(b, w.d, generator=gen, device=device, dtype=torch.float32)
    return _finish(x, w.torch_dtype)


def make_append_batch(w: Workload, centres: torch.Tensor, round_idx: int, seed: int = 0,
                      device="cpu"):
    """One streaming round's new entries: group ids drawn in proportion to the
    initial Zipf weights, embeddings from the same clustered generator."""
    gen = _gen(seed, 100 + 2 * round_idx, device)
    weights = torch.as_tensor(group_sizes(w), dtype=torch.float64, device=device)
    gid = torch.multinomial(weights, w.append_per_round, replacement=True, generator=gen)
    gid = gid.to(torch.int32)
    rows = make_rows(w, gid, centres, gen)
    return rows, gid


def to_numpy(x: torch.Tensor) -> np.ndarray:
    """Host numpy view for the oracle: float32 stays float32, bf16 becomes its
    uint16 bit pattern, int32 stays int32."""
    x = x.detach().contiguous()
    if x.dtype == torch.bfloat16:
        return x.view(torch.int16).cpu().numpy().view(np.uint16)
    return x.cpu().numpy()
