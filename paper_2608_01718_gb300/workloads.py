"""Seeded synthetic workloads for the two-stage lookahead lookup.

This module only draws inputs: cache entries (key embedding, lookahead-prefix embedding, prefix token ids) and
query batches (query embedding, the query's own k-token prefix embedding and ids). It holds none of the lookup's
arithmetic and is shared by the CUDA path's harness and by the oracle's tests.

The inputs stand in for what the paper's embedding model and draft LLM produce on its datasets (BGE-large 1024-d
or MiniLM 384-d embeddings, greedy k-token prefixes; §4.1 "LLMs and Embedding Models"). Those datasets are not
used here. The recipe:

* cluster centres: uniform random unit vectors;
* entry i: cluster a_i uniform; key = normalise(centre[a_i] + noise), where noise is Gaussian with expected norm
  ``cluster_sigma`` (per-component std ``cluster_sigma / sqrt(d)``); prefix embedding = an independent uniform unit
  vector; prefix ids uniform over the vocabulary;
* queries, shuffled within the batch:
  - near-duplicate (benign paraphrase): normalise(key_t + noise of norm ``near_sigma``), carrying entry t's
    prefix embedding (exact, or plus noise of norm ``near_prefix_sigma`` per model) and its ids (same greedy
    response prefix);
  - random: a uniform unit vector with a fresh prefix;
  - collision (the threat model's key collision): normalise(key_t + noise of norm ``coll_sigma``) with a fresh
    prefix embedding and fresh ids (a semantically distinct response);
  - mimic (ensemble workloads only): a collision whose response prefix is close to the victim's under the first
    embedding model and fresh under the others (the in-context attack whose prefix partly aligns, Figure 6);
* ensemble workloads hold one prefix embedding per model, concatenated in the prefix row, each a unit vector;
* targets t are uniform over the entries present at generation time, or Zipf(s) over a seeded permutation of them.

Noise is read as a vector whose expected norm is sigma. Read per component instead, a near-duplicate at d=384 and
sigma=0.05 would have cosine ~0.71 to its target and would never clear a 0.85 key threshold.

Everything is generated in fixed row chunks from counter-derived seeds, so that any chunk of the store can be
regenerated on its own (the oracle reads the store chunk by chunk for caches too large for host memory).
"""
from __future__ import annotations

import dataclasses
import hashlib
import math
from typing import Iterator

import torch

NEAR, RANDOM, COLLISION, MIMIC = 0, 1, 2, 3
CLASS_NAMES = {NEAR: "near-duplicate", RANDOM: "random", COLLISION: "collision", MIMIC: "mimic"}

# rows per generated store chunk; fixed so that chunk i is always the same rows
CHUNK_ROWS = 1 << 18


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n: int                      # entries in the cache (initial entries for the serve loop)
    d: int                      # embedding dimension (keys and prefix embeddings)
    k: int                      # lookahead window: prefix token ids per entry
    vocab: int
    clusters: int
    batch: int                  # queries per lookup
    mix: tuple                  # (near-duplicate, random, collision) fractions
    tau_c: float                # key (query) threshold
    tau_a: float                # lookahead (prefix) threshold
    top_c: int
    cluster_sigma: float = 0.15
    near_sigma: float = 0.05
    coll_sigma: float = 0.02
    key_dtype: str = "bf16"     # dtype the keys and prefix embeddings are handed to insert in
    zipf: float | None = None   # Zipf exponent over targets, None = uniform
    steps: int = 1              # serve-loop steps (batches); 1 = a single lookup
    seed: int = 20260801
    # Ensemble of m lookahead checks: one prefix embedding per model (these dimensions, concatenated in the
    # prefix row), each with its own threshold. None: one prefix embedding of dimension d checked with tau_a.
    prefix_dims: tuple | None = None
    tau_a_models: tuple | None = None
    near_prefix_sigma: float = 0.0   # noise norm on a near-duplicate's prefix embeddings (0: exact copies)

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def dims(self) -> tuple:
        return self.prefix_dims if self.prefix_dims is not None else (self.d,)

    @property
    def pd(self) -> int:
        """Length of a prefix row (all models' embeddings)."""
        return sum(self.dims)

    @property
    def store_bytes(self) -> int:
        return self.n * (2 * self.d + 2 * self.pd + 4 * self.k)


WORKLOADS = {
    # Tiny reference cache (fp32 keys rounded to bf16 at insert).
    "tiny-4k": Workload("tiny-4k", n=4096, d=384, k=8, vocab=32000, clusters=64, batch=64,
                        mix=(0.4, 0.3, 0.3), tau_c=0.85, tau_a=0.80, top_c=4, key_dtype="f32"),
    # Mid cache, bandwidth-bound scan (the headline benchmark workload).
    "mid-1m": Workload("mid-1m", n=1 << 20, d=768, k=16, vocab=128256, clusters=4096, batch=32,
                       mix=(0.5, 0.3, 0.2), tau_c=0.90, tau_a=0.80, top_c=8),
    # Large cache near HBM capacity, Zipf(1.1) popularity of near-duplicate targets.
    "large-16m": Workload("large-16m", n=1 << 24, d=1024, k=16, vocab=128256, clusters=4096, batch=128,
                          mix=(0.5, 0.3, 0.2), tau_c=0.90, tau_a=0.80, top_c=8, zipf=1.1),
    # Large query batch: a dense contraction on the tensor cores.
    "batch-4m": Workload("batch-4m", n=1 << 22, d=768, k=16, vocab=128256, clusters=4096, batch=8192,
                         mix=(0.6, 0.25, 0.15), tau_c=0.88, tau_a=0.80, top_c=16),
    # Streaming serve loop: 1000 batches, every miss appended.
    "serve-2m": Workload("serve-2m", n=1 << 21, d=768, k=32, vocab=128256, clusters=4096, batch=256,
                         mix=(0.45, 0.35, 0.2), tau_c=0.90, tau_a=0.80, top_c=8, steps=1000),
    # Ensemble of three lookahead checks (BGE-large, MiniLM and MPNet dimensions), with prefix-mimicking
    # collisions that only the ensemble rejects.
    "ensemble-1m": Workload("ensemble-1m", n=1 << 20, d=768, k=16, vocab=128256, clusters=4096, batch=32,
                            mix=(0.45, 0.25, 0.15, 0.15), tau_c=0.90, tau_a=0.70, top_c=8,
                            prefix_dims=(1024, 384, 768), tau_a_models=(0.70, 0.70, 0.70),
                            near_prefix_sigma=0.3),
}


def sub_seed(master: int, tag: str, index: int = 0) -> int:
    h = hashlib.sha256(f"{master}/{tag}/{index}".encode()).digest()
    return int.from_bytes(h[:8], "little") >> 2


def _gen(w: Workload, tag: str, index: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(sub_seed(w.seed, tag, index))
    return g


def _unit(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=1, keepdim=True)


def _unit_segments(x: torch.Tensor, dims: tuple) -> torch.Tensor:
    """Normalise each model's segment of a prefix row separately."""
    return torch.cat([_unit(part) for part in torch.split(x, list(dims), dim=1)], dim=1)


def centres(w: Workload, device="cpu") -> torch.Tensor:
    g = _gen(w, "centres", 0, device)
    return _unit(torch.randn((w.clusters, w.d), generator=g, device=device, dtype=torch.float32))


def _emb_dtype(w: Workload) -> torch.dtype:
    return torch.float32 if w.key_dtype == "f32" else torch.bfloat16


def store_chunk(w: Workload, index: int, device="cpu", cent: torch.Tensor | None = None) -> dict:
    """Rows [index*CHUNK_ROWS, min(n, (index+1)*CHUNK_ROWS)) of the initial store."""
    j0 = index * CHUNK_ROWS
    rows = min(w.n, j0 + CHUNK_ROWS) - j0
    if rows <= 0:
        raise IndexError(f"chunk {index} is past the {w.n}-row store")
    if cent is None:
        cent = centres(w, device)
    g = _gen(w, "store", index, device)
    cluster = torch.randint(0, w.clusters, (rows,), generator=g, device=device)
    noise = torch.randn((rows, w.d), generator=g, device=device) * (w.cluster_sigma / math.sqrt(w.d))
    key = _unit(cent[cluster] + noise)
    del noise
    prefix = _unit_segments(torch.randn((rows, w.pd), generator=g, device=device), w.dims)
    ids = torch.randint(0, w.vocab, (rows, w.k), generator=g, device=device, dtype=torch.int32)
    dt = _emb_dtype(w)
    return {"j0": j0, "key": key.to(dt), "prefix": prefix.to(dt), "ids": ids, "cluster": cluster}


def iter_store(w: Workload, device="cpu") -> Iterator[dict]:
    cent = centres(w, device)
    for index in range((w.n + CHUNK_ROWS - 1) // CHUNK_ROWS):
        yield store_chunk(w, index, device, cent)


def store_rows(w: Workload, rows: torch.Tensor, device="cpu") -> dict:
    """Regenerate selected rows of the initial store (chunk by chunk)."""
    rows = rows.to("cpu", torch.int64)
    out_key = torch.empty((len(rows), w.d), dtype=_emb_dtype(w), device=device)
    out_pre = torch.empty((len(rows), w.pd), dtype=_emb_dtype(w), device=device)
    out_ids = torch.empty((len(rows), w.k), dtype=torch.int32, device=device)
    if len(rows) == 0:
        return {"key": out_key, "prefix": out_pre, "ids": out_ids}
    cent = centres(w, device)
    chunk_of = rows // CHUNK_ROWS
    for index in torch.unique(chunk_of).tolist():
        sel = torch.nonzero(chunk_of == index).flatten()
        ch = store_chunk(w, index, device, cent)
        local = (rows[sel] - ch["j0"]).to(device)
        sel_d = sel.to(device)
        out_key[sel_d] = ch["key"][local]
        out_pre[sel_d] = ch["prefix"][local]
        out_ids[sel_d] = ch["ids"][local]
    return {"key": out_key, "prefix": out_pre, "ids": out_ids}


def class_counts(w: Workload) -> tuple:
    """(near-duplicate, random, collision[, mimic]) query counts of a batch."""
    near = min(int(round(w.batch * w.mix[0])), w.batch)
    coll = min(int(round(w.batch * w.mix[2])), w.batch - near)
    if len(w.mix) > 3:
        mimic = min(int(round(w.batch * w.mix[3])), w.batch - near - coll)
        return near, w.batch - near - coll - mimic, coll, mimic
    return near, w.batch - near - coll, coll


def query_plan(w: Workload, step: int = 0, n_entries: int | None = None) -> dict:
    """Class and target entry of every query of batch ``step`` (drawn on the CPU: small)."""
    n_entries = w.n if n_entries is None else n_entries
    g = _gen(w, "plan", step, "cpu")
    counts = class_counts(w)
    near, rand, coll = counts[:3]
    mimic = counts[3] if len(counts) > 3 else 0
    classes = torch.tensor([NEAR] * near + [RANDOM] * rand + [COLLISION] * coll + [MIMIC] * mimic,
                           dtype=torch.int64)
    classes = classes[torch.randperm(w.batch, generator=g)]
    if w.zipf is None:
        target = torch.randint(0, max(n_entries, 1), (w.batch,), generator=g)
    else:
        # Zipf(s) over ranks 1..n, mapped to entries by a seeded affine permutation of [0, n)
        ranks = torch.arange(1, n_entries + 1, dtype=torch.float64)
        cdf = torch.cumsum(ranks.pow(-w.zipf), 0)
        cdf /= cdf[-1].clone()
        u = torch.rand((w.batch,), generator=g, dtype=torch.float64)
        r = torch.searchsorted(cdf, u).clamp_(max=n_entries - 1)
        a = int(torch.randint(1, 1 << 30, (1,), generator=g)) | 1
        while math.gcd(a, n_entries) != 1:
            a += 2
        b = int(torch.randint(0, n_entries, (1,), generator=g))
        target = (r * a + b) % n_entries
    target = torch.where(classes == RANDOM, torch.full_like(target, -1), target)
    return {"class": classes, "target": target}


def make_queries(w: Workload, plan: dict, step: int = 0, device="cpu", target_rows: dict | None = None) -> dict:
    """Query embeddings, prefix embeddings (bf16) and prefix ids (int32) for one batch."""
    B = w.batch
    cls = plan["class"].to(device)
    tgt = plan["target"].clone()
    if target_rows is None:
        target_rows = store_rows(w, tgt.clamp(min=0), device)
    g = _gen(w, "queries", step, device)
    base = target_rows["key"].to(torch.float32)
    noise = torch.randn((B, w.d), generator=g, device=device)
    rnd = torch.randn((B, w.d), generator=g, device=device)
    fresh_pre = _unit_segments(torch.randn((B, w.pd), generator=g, device=device), w.dims).to(torch.bfloat16)
    fresh_ids = torch.randint(0, w.vocab, (B, w.k), generator=g, device=device, dtype=torch.int32)
    scale = torch.where(cls == NEAR, w.near_sigma, w.coll_sigma).to(torch.float32)[:, None] / math.sqrt(w.d)
    q = torch.where((cls == RANDOM)[:, None], rnd, base + noise * scale)
    q = _unit(q).to(torch.bfloat16)
    near = (cls == NEAR)[:, None]
    tpre = target_rows["prefix"].to(torch.float32)
    if w.near_prefix_sigma > 0:
        # a paraphrase's response prefix: the target's prefix embeddings plus noise of the given norm per model
        pn = torch.randn((B, w.pd), generator=g, device=device)
        seg_scale = torch.cat([torch.full((dim,), w.near_prefix_sigma / math.sqrt(dim), device=device)
                               for dim in w.dims])
        tpre = _unit_segments(tpre + pn * seg_scale, w.dims)
    pre = torch.where(near, tpre.to(torch.bfloat16), fresh_pre)
    # a prefix-mimicking collision: close to the victim's response prefix under the first model only
    d0 = w.dims[0]
    mimic = (cls == MIMIC)[:, None]
    pre[:, :d0] = torch.where(mimic, tpre[:, :d0].to(torch.bfloat16), pre[:, :d0])
    ids = torch.where(near, target_rows["ids"], fresh_ids)
    return {"emb": q.contiguous(), "prefix": pre.contiguous(), "ids": ids.contiguous(),
            "class": plan["class"].clone(), "target": plan["target"].clone()}


def batch(w: Workload, step: int = 0, device="cpu", n_entries: int | None = None) -> dict:
    plan = query_plan(w, step, n_entries)
    return make_queries(w, plan, step, device)


def bf16_bits(t: torch.Tensor):
    """Host numpy view of a bf16 tensor's bit patterns (uint16): the exact bytes both sides read."""
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view("uint16")


def f32_array(t: torch.Tensor):
    return t.detach().to("cpu", torch.float32).contiguous().numpy()


def benign_pairs(n: int, d: int, sigma: float, seed: int = 20260801, device="cpu"):
    """n benign paraphrase pairs (x, x'): x a uniform unit vector and x' = normalise(x + noise of norm sigma),
    both bf16 [n x d]. Stand-ins for the embeddings of the paper's 500 paraphrase pairs used to calibrate the
    thresholds (App. A.2)."""
    g = torch.Generator(device=device)
    g.manual_seed(sub_seed(seed, f"benign/{n}/{d}/{sigma}", 0))
    x = _unit(torch.randn((n, d), generator=g, device=device))
    y = _unit(x + torch.randn((n, d), generator=g, device=device) * (sigma / math.sqrt(d)))
    return x.to(torch.bfloat16).contiguous(), y.to(torch.bfloat16).contiguous()


def hyperplanes(bits: int, d: int, seed: int = 20260801, device="cpu") -> torch.Tensor:
    """Random hyperplanes of the SimHash index, bf16 [bits x d] with standard normal entries."""
    g = torch.Generator(device=device)
    g.manual_seed(sub_seed(seed, f"hyperplanes/{bits}/{d}", 0))
    return torch.randn((bits, d), generator=g, device=device).to(torch.bfloat16).contiguous()


def lsh_radius(tau_c: float, bits: int, z: float = 4.0) -> int:
    """A Hamming radius that keeps an entry at the key threshold with probability about Phi(z): the number of
    differing bits at angle arccos(tau_c) is Binomial(bits, theta / pi)."""
    theta = math.acos(max(-1.0, min(1.0, tau_c)))
    p = theta / math.pi
    return min(bits, int(math.ceil(bits * p + z * math.sqrt(bits * p * (1 - p)))))


def draft_probabilities(batch: int, k: int, seed: int = 20260801, device="cpu"):
    """Stand-ins for the target's and the draft's probabilities of each of the k draft tokens, [batch x k] fp32:
    correlated uniforms, so that acceptance runs of every length occur."""
    g = torch.Generator(device=device)
    g.manual_seed(sub_seed(seed, f"draft/{batch}/{k}", 0))
    pg = torch.rand((batch, k), generator=g, device=device)
    pf = (pg + 0.2 * torch.randn((batch, k), generator=g, device=device) + 0.3).clamp(0.0, 1.0)
    return pf.contiguous(), pg.contiguous()
