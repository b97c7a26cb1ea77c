"""Seeded synthetic inputs for the paged tensor store.

This module is shared by the CPU oracle (``oracle/``) and by the GPU path's
tests and benchmark. It holds random draws and workload shapes only: no page
placement, copying, casting, eviction or compaction arithmetic lives here.

The paper's workloads are production T2I traces and real Flux/DiT models
(§8.1 Setup, Table 1); none of them is available, so the five workloads below
stand in for them with the shapes of a Flux-style workflow (§2.1, §5.1):

* ``tiny``       -- 64 MiB pool, 64 KiB pages, 32 + 8 uint8 objects.
* ``handoff``    -- 8 GiB pool, 2 MiB pages, per-request text embeddings,
                    pooled embeddings, latents and decoded images (§5.2).
* ``weights``    -- 40 GiB pool, 2 MiB pages, bf16 weights of a 57-block DiT
                    (hidden 3072, MLP 12288), restored from pinned host (§5.1).
* ``adapters``   -- 16 GiB pool, 256 KiB pages, 512 LoRA sets, Zipf(1.1)
                    popularity, LRU eviction (§5.3).
* ``compaction`` -- 64 GiB pool, 2 MiB pages, fragmented by a seeded trace of
                    100,000 alloc/free ops, then compacted to 48 GiB.

bf16 inputs are produced by keeping the upper 16 bits of an fp32 draw
(round toward zero). That is only a way to obtain bf16 numbers with the stated
distribution; the store's own fp32->bf16 round-to-nearest-even cast is not
used to make any input.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

KiB = 1024
MiB = 1024 * KiB
GiB = 1024 * MiB


def rng(seed: int, *stream: int) -> np.random.Generator:
    """A PCG64 generator for (seed, stream...) -- independent streams per use."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), *map(int, stream)])))


def log_uniform_sizes(g: np.random.Generator, k: int, lo: int, hi: int) -> np.ndarray:
    """floor(exp(U(ln lo, ln hi))) bytes, k draws."""
    return np.floor(np.exp(g.uniform(math.log(lo), math.log(hi), int(k)))).astype(np.int64)


def bf16_bits_from_f32(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of fp32 numbers by truncation (input generation only)."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


# --------------------------------------------------------------------------
# tiny: 64 MiB pool, 64 KiB pages
# --------------------------------------------------------------------------
TINY = dict(pool_bytes=64 * MiB, page_bytes=64 * KiB, n_first=32, n_more=8, lo=1 * KiB, hi=2 * MiB)


def tiny_objects(seed: int = 0, n_first: int = 32, n_more: int = 8, lo: int = 1 * KiB, hi: int = 2 * MiB):
    """Two lists of uint8 arrays: the first ``n_first`` objects and ``n_more``
    objects drawn afterwards from the same stream. Sizes are log-uniform in
    [lo, hi), bytes uniform in [0, 256)."""
    g = rng(seed, 1)

    def draw(k):
        return [g.integers(0, 256, int(n), dtype=np.uint8) for n in log_uniform_sizes(g, k, lo, hi)]

    first = draw(n_first)
    more = draw(n_more)
    return first, more


def tiny_freed_indices(n_first: int = 32) -> list[int]:
    """"Free every third object": indices i with i % 3 == 2."""
    return [i for i in range(n_first) if i % 3 == 2]


# --------------------------------------------------------------------------
# handoff: T2I intermediates, 8 GiB pool, 2 MiB pages
# --------------------------------------------------------------------------
HANDOFF = dict(pool_bytes=8 * GiB, page_bytes=2 * MiB, requests=64, batch_sizes=(1, 4, 8))

# dtype tags carried by the store's directory (metadata only)
DTYPE_U8, DTYPE_BF16, DTYPE_F16, DTYPE_F32 = 0, 1, 2, 3
ITEMSIZE = {DTYPE_U8: 1, DTYPE_BF16: 2, DTYPE_F16: 2, DTYPE_F32: 4}


@dataclass(frozen=True)
class TensorSpec:
    name: str
    dtype_tag: int
    shape: tuple

    @property
    def numel(self) -> int:
        return int(np.prod(self.shape, dtype=np.int64))

    @property
    def nbytes(self) -> int:
        return self.numel * ITEMSIZE[self.dtype_tag]


def handoff_specs(B: int, text_len: int = 512, text_dim: int = 4096, pooled_dim: int = 768,
                  lat_c: int = 16, lat_hw: int = 128, img_hw: int = 1024) -> list[TensorSpec]:
    """The four intermediates one request hands from model to model (§2.1, §5.2):
    text embeddings, pooled embeddings, latents and the decoded image."""
    return [
        TensorSpec("text", DTYPE_BF16, (B, text_len, text_dim)),
        TensorSpec("pooled", DTYPE_BF16, (B, pooled_dim)),
        TensorSpec("latents", DTYPE_F32, (B, lat_c, lat_hw, lat_hw)),
        TensorSpec("image", DTYPE_F16, (B, 3, img_hw, img_hw)),
    ]


def handoff_cast_index() -> int:
    """Position of the latents in :func:`handoff_specs`: got with the fp32->bf16 cast."""
    return 2


def handoff_request(seed: int, r: int, specs: list[TensorSpec]) -> list[np.ndarray]:
    """Host arrays (uint16 bf16 bits / float32 / float16) for request ``r``:
    text and pooled N(0,1) as bf16, latents N(0,1) fp32, image U[-1,1] fp16."""
    g = rng(seed, 2, r)
    out = []
    for s in specs:
        if s.dtype_tag == DTYPE_BF16:
            out.append(bf16_bits_from_f32(g.standard_normal(s.numel, dtype=np.float32)).reshape(s.shape))
        elif s.dtype_tag == DTYPE_F32:
            out.append(g.standard_normal(s.numel, dtype=np.float32).reshape(s.shape))
        elif s.dtype_tag == DTYPE_F16:
            out.append(g.uniform(-1.0, 1.0, s.numel).astype(np.float16).reshape(s.shape))
        else:
            out.append(g.integers(0, 256, s.numel, dtype=np.uint8).reshape(s.shape))
    return out


def handoff_request_torch(seed: int, r: int, specs: list[TensorSpec], device):
    """Same distributions as :func:`handoff_request`, drawn by torch's
    generator on ``device`` (fast for the full-size benchmark; values differ
    from the numpy draw)."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + 7919 * int(r)) & 0x7FFFFFFFFFFFFFFF)
    out = []
    for s in specs:
        if s.dtype_tag == DTYPE_BF16:
            x = torch.randn(s.shape, generator=g, device=device, dtype=torch.float32)
            out.append((x.view(torch.int32) >> 16).to(torch.int16).view(torch.bfloat16))
        elif s.dtype_tag == DTYPE_F32:
            out.append(torch.randn(s.shape, generator=g, device=device, dtype=torch.float32))
        elif s.dtype_tag == DTYPE_F16:
            x = torch.rand(s.shape, generator=g, device=device, dtype=torch.float32) * 2.0 - 1.0
            out.append(x.to(torch.float16))
        else:
            out.append(torch.randint(0, 256, s.shape, generator=g, device=device, dtype=torch.uint8))
    return out


# --------------------------------------------------------------------------
# weights: 57-block DiT, bf16, ~11.84 B parameters
# --------------------------------------------------------------------------
WEIGHTS = dict(pool_bytes=40 * GiB, page_bytes=2 * MiB)


@dataclass(frozen=True)
class WeightSpec:
    name: str
    shape: tuple
    block: int

    @property
    def numel(self) -> int:
        return int(np.prod(self.shape, dtype=np.int64))

    @property
    def nbytes(self) -> int:
        return 2 * self.numel


def dit_weight_specs(hidden: int = 3072, mlp: int = 12288, head_dim: int = 128,
                     n_double: int = 19, n_single: int = 38) -> list[WeightSpec]:
    """Tensor list of a Flux-style DiT: ``n_double`` two-stream blocks (16
    tensors per stream) then ``n_single`` single-stream blocks (14 tensors)."""
    h, m = hidden, mlp
    out: list[WeightSpec] = []
    for b in range(n_double):
        for st in ("img", "txt"):
            p = f"double{b}.{st}."
            for nm in ("q", "k", "v", "o"):
                out += [WeightSpec(p + nm + ".w", (h, h), b), WeightSpec(p + nm + ".b", (h,), b)]
            out += [WeightSpec(p + "fc1.w", (m, h), b), WeightSpec(p + "fc1.b", (m,), b),
                    WeightSpec(p + "fc2.w", (h, m), b), WeightSpec(p + "fc2.b", (h,), b),
                    WeightSpec(p + "mod.w", (6 * h, h), b), WeightSpec(p + "mod.b", (6 * h,), b),
                    WeightSpec(p + "q_norm", (head_dim,), b), WeightSpec(p + "k_norm", (head_dim,), b)]
    for j in range(n_single):
        b = n_double + j
        p = f"single{j}."
        for nm in ("q", "k", "v"):
            out += [WeightSpec(p + nm + ".w", (h, h), b), WeightSpec(p + nm + ".b", (h,), b)]
        out += [WeightSpec(p + "mlp_in.w", (m, h), b), WeightSpec(p + "mlp_in.b", (m,), b),
                WeightSpec(p + "out.w", (h, h + m), b), WeightSpec(p + "out.b", (h,), b),
                WeightSpec(p + "mod.w", (3 * h, h), b), WeightSpec(p + "mod.b", (3 * h,), b),
                WeightSpec(p + "q_norm", (head_dim,), b), WeightSpec(p + "k_norm", (head_dim,), b)]
    return out


def block_layout(specs, align: int = 256):
    """Per-block contiguous buffers: for each block, (total bytes, [(spec index,
    byte offset)]) with every tensor ``align``-aligned inside its block buffer
    in list order."""
    blocks: dict[int, list] = {}
    sizes: dict[int, int] = {}
    for i, s in enumerate(specs):
        off = sizes.get(s.block, 0)
        off = (off + align - 1) // align * align
        blocks.setdefault(s.block, []).append((i, off))
        sizes[s.block] = off + s.nbytes
    return [(sizes[b], blocks[b]) for b in sorted(blocks)]


def weight_values_torch(seed: int, index: int, spec: WeightSpec, device, std: float = 0.02):
    """N(0, std) bf16 values (upper 16 bits of an fp32 draw) seeded per tensor
    with ``seed + index``, drawn by torch on ``device``."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(int(seed) + int(index))
    x = torch.randn(spec.numel, generator=g, device=device, dtype=torch.float32) * std
    return (x.view(torch.int32) >> 16).to(torch.int16).view(torch.bfloat16)


# --------------------------------------------------------------------------
# adapters: 512 LoRA sets on the same DiT, Zipf(1.1) popularity
# --------------------------------------------------------------------------
ADAPTERS = dict(pool_bytes=16 * GiB, page_bytes=256 * KiB, n_sets=512, n_calls=10_000, window=256,
                ranks=(8, 16, 32, 64), zipf_s=1.1)


def lora_projections(hidden: int = 3072, mlp: int = 12288, n_double: int = 19, n_single: int = 38):
    """(block, in_features, out_features) of every adapted projection: per
    double-block stream q, k, v, o, fc1, fc2; per single block q, k, v,
    mlp_in, out. 418 projections for the default DiT."""
    h, m = hidden, mlp
    out = []
    for b in range(n_double):
        for _st in range(2):
            out += [(b, h, h)] * 4 + [(b, h, m), (b, m, h)]
    for j in range(n_single):
        b = n_double + j
        out += [(b, h, h)] * 3 + [(b, h, m), (b, h + m, h)]
    return out


def lora_objects(rank: int, projections=None):
    """Objects of one LoRA set in order: for each projection, A [r, in] then
    B [out, r], bf16. Returns a list of (block, nbytes)."""
    projections = lora_projections() if projections is None else projections
    objs = []
    for (b, fin, fout) in projections:
        objs.append((b, 2 * rank * fin))
        objs.append((b, 2 * fout * rank))
    return objs


def lora_ranks(seed: int, n_sets: int = 512, ranks=(8, 16, 32, 64)) -> np.ndarray:
    g = rng(seed, 4, 1)
    return np.asarray(ranks, dtype=np.int64)[g.integers(0, len(ranks), n_sets)]


def zipf_ranks(g: np.random.Generator, k: int, n: int, s: float) -> np.ndarray:
    """k draws of a rank in 1..n with P(rank) proportional to rank**-s."""
    w = np.arange(1, n + 1, dtype=np.float64) ** (-float(s))
    cdf = np.cumsum(w / w.sum())
    cdf[-1] = 1.0
    return np.searchsorted(cdf, g.random(int(k)), side="right") + 1


def adapter_calls(seed: int, n_calls: int = 10_000, n_sets: int = 512, n_objects: int = 836,
                  window: int = 256, s: float = 1.1):
    """(set ids, window starts) of the get_batch calls: a Zipf(s) rank mapped
    to a set through a seeded permutation, and a window start uniform in
    [0, n_objects - window]."""
    g = rng(seed, 4, 2)
    perm = g.permutation(n_sets)
    ranks = zipf_ranks(g, n_calls, n_sets, s)
    sets = perm[ranks - 1]
    starts = g.integers(0, n_objects - window + 1, n_calls)
    return sets.astype(np.int64), starts.astype(np.int64)


def lora_bank_offsets(seed: int, set_bytes: np.ndarray, bank_bytes: int, align: int = 256) -> np.ndarray:
    """Each set's contents are the bank window [off, off + set_bytes): a seeded
    ``align``-aligned offset per set (so set contents differ between sets)."""
    g = rng(seed, 4, 3)
    room = (bank_bytes - np.asarray(set_bytes, dtype=np.int64)) // align
    if np.any(room < 0):
        raise ValueError("bank smaller than a set")
    return (np.floor(g.random(len(room)) * (room + 1)).astype(np.int64)) * align


def lora_bank_torch(seed: int, bank_bytes: int, device, std: float = 0.01):
    """The adapter value bank: N(0, std) bf16 values as raw bytes on ``device``."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 7 + 4)
    x = torch.randn(bank_bytes // 2, generator=g, device=device, dtype=torch.float32) * std
    return (x.view(torch.int32) >> 16).to(torch.int16).view(torch.uint8)


# --------------------------------------------------------------------------
# compaction: 64 GiB pool, 2 MiB pages, seeded alloc/free trace
# --------------------------------------------------------------------------
COMPACTION = dict(pool_bytes=64 * GiB, page_bytes=2 * MiB, n_ops=100_000, lo=4 * KiB, hi=512 * MiB,
                  p_free=0.5, settle_frac=0.5, limit_bytes=48 * GiB)


@dataclass
class Trace:
    ops: list            # ("alloc", k, nbytes) | ("free", k); k = the trace's object number
    sizes: dict          # k -> nbytes
    survivors: list      # object numbers live at the end, ascending
    skipped: int         # allocs that did not fit and were skipped
    n_ops: int


def compaction_trace(seed: int, total_pages: int, page_bytes: int, n_ops: int = 100_000,
                     lo: int = 4 * KiB, hi: int = 512 * MiB, p_free: float = 0.5,
                     settle_frac: float = 0.5) -> Trace:
    """The fragmenting alloc/free sequence, defined on page demand
    ceil(nbytes / page_bytes) against ``total_pages``:

    1. allocate until the first allocation that does not fit;
    2. then, until ``n_ops`` operations (phase 1 included) have been drawn:
       with probability ``p_free`` free a uniformly chosen live object, else
       allocate a log-uniform size; an allocation that does not fit is skipped;
    3. settle: free uniformly chosen live objects until at most
       ``settle_frac`` of the pages are in use.
    """
    g = rng(seed, 5)
    need = lambda n: -(-int(n) // page_bytes)  # page demand of an object
    used = 0
    live: list[int] = []
    sizes: dict[int, int] = {}
    ops: list = []
    skipped = 0
    k = 0
    drawn = 0
    while drawn < n_ops:  # phase 1
        n = int(log_uniform_sizes(g, 1, lo, hi)[0])
        drawn += 1
        if used + need(n) > total_pages:
            skipped += 1
            break
        sizes[k] = n
        ops.append(("alloc", k, n))
        live.append(k)
        used += need(n)
        k += 1
    while drawn < n_ops:  # phase 2
        drawn += 1
        if g.random() < p_free:
            if not live:
                continue
            j = int(g.random() * len(live))
            victim = live.pop(j)
            ops.append(("free", victim))
            used -= need(sizes[victim])
        else:
            n = int(log_uniform_sizes(g, 1, lo, hi)[0])
            if used + need(n) > total_pages:
                skipped += 1
                continue
            sizes[k] = n
            ops.append(("alloc", k, n))
            live.append(k)
            used += need(n)
            k += 1
    while live and used > settle_frac * total_pages:  # phase 3
        j = int(g.random() * len(live))
        victim = live.pop(j)
        ops.append(("free", victim))
        used -= need(sizes[victim])
    return Trace(ops=ops, sizes=sizes, survivors=sorted(live), skipped=skipped, n_ops=n_ops)


def object_bytes(seed: int, k: int, nbytes: int) -> np.ndarray:
    """Uniform random bytes of object ``k`` (numpy; for small objects)."""
    g = rng(seed, 6, k)
    return g.integers(0, 256, int(nbytes), dtype=np.uint8)
