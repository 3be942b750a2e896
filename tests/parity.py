"""Helpers for the GPU-vs-oracle parity tests: build a device cache from a workload, run lookups through the C ABI,
feed the oracle the same bytes, and compare.

The comparison rules follow from the arithmetic. The GPU accumulates bf16 products in fp32; the oracle sums
them exactly in fp64. For unit vectors with d <= 8192, the fp32 error is far below TOL = 2e-3:
  * scores (key, prefix; per candidate) agree within TOL everywhere;
  * status, entry id, token matches and candidate count agree exactly for every query whose oracle decision
    margin is >= TOL (the others are counted and reported; for them a HIT must still pass both checks
    within TOL);
  * a candidate id must agree exactly unless its score is within TOL of a neighbour in the oracle's order (a
    near-tie), in which case it must be one of the oracle's tied entries.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

import oracle
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

TOL = 2e-3


def new_cache(w: wl.Workload, stage1: int, device: int = 0, capacity: int | None = None, **kw) -> L.LaCache:
    if w.prefix_dims is not None:
        kw.setdefault("prefix_dims", w.prefix_dims)
        kw.setdefault("tau_a_models", w.tau_a_models)
    return L.LaCache(w.d, w.k, capacity or w.n, w.tau_c, w.tau_a, w.top_c, max_batch=kw.pop("max_batch", w.batch),
                     device=device, stage1=stage1, **kw)


def fill(cache: L.LaCache, w: wl.Workload, device="cuda") -> None:
    dtype = L.LACACHE_F32 if w.key_dtype == "f32" else L.LACACHE_BF16
    for ch in wl.iter_store(w, device):
        cache.insert(ch["key"], ch["prefix"], ch["ids"], dtype)
    torch.cuda.synchronize()


def _bits(t: torch.Tensor, f32: bool):
    return oracle.round_to_bf16(wl.f32_array(t)) if f32 else wl.bf16_bits(t)


def oracle_store(w: wl.Workload, device="cuda") -> oracle.Store:
    """The whole initial store as host bf16 bit patterns (for caches that fit host memory)."""
    keys, pres, ids = [], [], []
    f32 = w.key_dtype == "f32"
    for ch in wl.iter_store(w, device):
        keys.append(_bits(ch["key"], f32))
        pres.append(_bits(ch["prefix"], f32))
        ids.append(ch["ids"].cpu().numpy())
    return oracle.Store.of(np.concatenate(keys), np.concatenate(pres), np.concatenate(ids))


def oracle_queries(q: dict, rows=None) -> dict:
    sel = slice(None) if rows is None else rows
    return {"emb": wl.bf16_bits(q["emb"][sel]), "prefix": wl.bf16_bits(q["prefix"][sel]),
            "ids": q["ids"][sel].cpu().numpy()}


def params(w: wl.Workload, check_mode=oracle.CHECK_EMB, token_match_min=None) -> oracle.Params:
    # the GPU compares fp32 scores with the fp32 thresholds it was given; the oracle takes the same values
    f32 = lambda x: float(np.float32(x))
    if w.prefix_dims is not None:
        return oracle.Params(f32(w.tau_c), 0.0, w.top_c, check_mode, token_match_min, prefix_dims=w.prefix_dims,
                             tau_a_models=tuple(f32(t) for t in w.tau_a_models))
    return oracle.Params(f32(w.tau_c), f32(w.tau_a), w.top_c, check_mode, token_match_min)


def gpu_lookup(cache: L.LaCache, q: dict) -> dict:
    out = cache.lookup(q["emb"], q["prefix"], q["ids"])
    torch.cuda.synchronize()
    cache.sync()
    return {k: v.cpu().numpy() for k, v in out.items()}


@dataclasses.dataclass
class Report:
    queries: int = 0
    band: int = 0
    literal_band: int = 0
    exact: int = 0
    hits: int = 0
    rejects: int = 0
    misses: int = 0
    near_ties: int = 0

    def add(self, other: "Report") -> None:
        for f in dataclasses.fields(self):
            setattr(self, f.name, getattr(self, f.name) + getattr(other, f.name))


def log_report(name: str, rep: Report) -> None:
    """One line per parity case (visible with pytest -s): what was compared and what fell in the margin band."""
    print(f"PARITY {name}: queries={rep.queries} exact={rep.exact} band={rep.band} literal_band={rep.literal_band} "
          f"hits={rep.hits} rejects={rep.rejects} misses={rep.misses} near_ties={rep.near_ties}", flush=True)


def _close(a, b, tol=TOL) -> bool:
    if np.isnan(a) and np.isnan(b):
        return True
    if np.isinf(a) or np.isinf(b):
        return a == b
    return abs(float(a) - float(b)) <= tol


def compare(gpu: dict, res: oracle.Result, p: oracle.Params, rows=None, pair_scores=None) -> Report:
    """Check a GPU lookup against the oracle's result for the same queries (``rows`` selects GPU rows).

    ``pair_scores(b, j)`` -> (s, r) gives the oracle's exact scores of query b against entry j, used to validate a
    HIT inside the margin band.
    """
    idx = np.arange(len(res.status)) if rows is None else np.asarray(rows)
    rep = Report(queries=len(idx))
    rep.literal_band = int(np.sum(res.literal_margin < TOL))
    for b, g in enumerate(idx):
        st = int(gpu["status"][g])
        assert st in (oracle.MISS_KEY, oracle.HIT, oracle.REJECT), f"query {g}: status {st}"
        in_band = res.margin[b] < TOL
        if in_band:
            rep.band += 1
            if st == oracle.HIT and pair_scores is not None:
                s, r, m, k = pair_scores(b, int(gpu["entry_id"][g]))
                assert s >= p.tau_c - TOL, f"query {g}: in-band HIT fails the key check"
                if p.check_mode in (oracle.CHECK_EMB, oracle.CHECK_BOTH) and p.prefix_dims is None:
                    assert r >= p.tau_a - TOL, f"query {g}: in-band HIT fails the lookahead check"
                if p.check_mode in (oracle.CHECK_TOKENS, oracle.CHECK_BOTH):
                    assert m >= (p.token_match_min or k), f"query {g}: in-band HIT fails the token check"
            continue
        msg = f"query {g} (oracle row {b})"
        assert st == res.status[b], f"{msg}: status {st} vs oracle {res.status[b]}"
        assert gpu["entry_id"][g] == res.entry_id[b], f"{msg}: entry {gpu['entry_id'][g]} vs {res.entry_id[b]}"
        assert _close(gpu["key_score"][g], res.key_score[b]), \
            f"{msg}: key score {gpu['key_score'][g]} vs {res.key_score[b]}"
        assert _close(gpu["prefix_score"][g], res.prefix_score[b]), f"{msg}: prefix score"
        assert gpu["token_matches"][g] == res.token_matches[b], f"{msg}: token matches"
        if "prefix_scores" in gpu:
            for h in range(res.prefix_scores.shape[1]):
                assert _close(gpu["prefix_scores"][g, h], res.prefix_scores[b, h]), f"{msg}: model {h} score"
        if res.list_margin[b] >= TOL:
            assert gpu["n_cand"][g] == res.n_cand[b], f"{msg}: n_cand {gpu['n_cand'][g]} vs {res.n_cand[b]}"
        if "cand_id" in gpu:
            _compare_candidates(gpu, res, g, b, rep, msg, p)
        rep.exact += 1
        rep.hits += st == oracle.HIT
        rep.rejects += st == oracle.REJECT
        rep.misses += st == oracle.MISS_KEY
    return rep


def pair_scores_fn(store: oracle.Store, oq: dict):
    """(s, r, m, k) of oracle query row b against entry j, from the host bytes through the oracle's own stages."""
    def f(b, j):
        kc = oracle.KeyCheck(oq["emb"][b:b + 1], -np.inf)
        kc.add_rows(store.key[j:j + 1], j)
        r, m = oracle.lookahead(oq["prefix"][b], oq["ids"][b], store.prefix[j:j + 1], store.ids[j:j + 1])
        return float(kc.best[0]), float(r[0]), int(m[0]), store.ids.shape[1]
    return f


def _pass_settled(res, b, i, p) -> bool:
    """Candidate i's pass bit is not within the tolerance of flipping (every threshold it uses is clear)."""
    if p.check_mode == oracle.CHECK_TOKENS:
        return True
    taus = p.tau_a_models if p.prefix_dims is not None else (p.tau_a,)
    return all(abs(res.cand_prefix_scores[b, i, h] - t) >= TOL for h, t in enumerate(taus))


def _compare_candidates(gpu, res, g, b, rep, msg, p):
    nc = int(res.n_cand[b])
    c = res.cand_id.shape[1]
    ng = int(gpu["n_cand"][g])
    o_ids = list(res.cand_id[b, :nc])
    o_scores = list(res.cand_score[b, :nc])
    if res.next_id[b] >= 0:
        o_ids.append(int(res.next_id[b]))
        o_scores.append(float(res.next_score[b]))
    for i in range(min(nc, ng)):
        gid, gs = int(gpu["cand_id"][g, i]), float(gpu["cand_score"][g, i])
        assert abs(gs - o_scores[i]) <= TOL, f"{msg}: candidate {i} score {gs} vs {o_scores[i]}"
        tied = (i > 0 and o_scores[i - 1] - o_scores[i] < TOL) or \
               (i + 1 < len(o_scores) and o_scores[i] - o_scores[i + 1] < TOL)
        if not tied:
            assert gid == o_ids[i], f"{msg}: candidate {i} id {gid} vs {o_ids[i]}"
            assert _close(gpu["cand_prefix_score"][g, i], res.cand_prefix_score[b, i]), f"{msg}: cand r {i}"
            assert gpu["cand_matches"][g, i] == res.cand_matches[b, i], f"{msg}: cand m {i}"
            if "cand_pass" in gpu and _pass_settled(res, b, i, p):
                assert bool(gpu["cand_pass"][g, i]) == bool(res.cand_pass[b, i]), f"{msg}: cand pass {i}"
            if "cand_prefix_scores" in gpu:
                for h in range(res.cand_prefix_scores.shape[2]):
                    assert _close(gpu["cand_prefix_scores"][g, i, h], res.cand_prefix_scores[b, i, h]), \
                        f"{msg}: cand {i} model {h} score"
        else:
            rep.near_ties += 1
            pos = [k for k, j in enumerate(o_ids) if j == gid]
            assert pos and abs(o_scores[pos[0]] - gs) <= TOL, f"{msg}: tied candidate {gid} not in oracle order"
    for i in range(ng, c):
        assert gpu["cand_id"][g, i] == -1 and np.isnan(gpu["cand_score"][g, i])
        if "cand_pass" in gpu:
            assert gpu["cand_pass"][g, i] == 0


class StreamedOracle:
    """The oracle for caches too large for host memory: the store streams through it chunk by chunk.

    Each generated chunk is inserted into the GPU cache and its key bytes go through the oracle's block-wise key
    check (A_q is a union over blocks). The prefix rows and ids of the entries stage 2 and the decision margin
    may need (every entry of each A_q: the margin of a rejection looks past the candidate cut) are then
    regenerated from the generator, never read back from the device. With no cache the store is generated on
    `device` only for the oracle. With `lsh` = (hyperplane bits, radius) the cache search is the SimHash index
    (oracle.LshKeyCheck), and `ambiguous` marks the sampled queries that ambiguous signature bits could change.
    """

    def __init__(self, w: wl.Workload, q: dict, sample, p: oracle.Params, lsh=None):
        self.w, self.q, self.p = w, q, p
        self.sample = np.asarray(sample)
        self.oq = oracle_queries(q, torch.as_tensor(self.sample))
        self.lk = oracle.LshKeyCheck(self.oq["emb"], p.tau_c, *lsh) if lsh is not None else None
        self.kc = self.lk.kc if self.lk is not None else oracle.KeyCheck(self.oq["emb"], p.tau_c)
        self.device = "cuda"

    @property
    def ambiguous(self):
        return self.lk.ambiguous if self.lk is not None else np.zeros(len(self.sample), dtype=bool)

    def fill(self, cache: L.LaCache | None, device="cuda") -> None:
        self.device = device
        dtype = L.LACACHE_F32 if self.w.key_dtype == "f32" else L.LACACHE_BF16
        for ch in wl.iter_store(self.w, device):
            if cache is not None:
                cache.insert(ch["key"], ch["prefix"], ch["ids"], dtype)
            (self.lk or self.kc).add_rows(_bits(ch["key"], self.w.key_dtype == "f32"), ch["j0"])
            del ch
        if device != "cpu":
            torch.cuda.synchronize()

    def result(self) -> oracle.Result:
        need = set()
        for b in range(len(self.sample)):
            _, j = self.kc.above(b)
            need.update(int(x) for x in j)
        ids = np.array(sorted(need), dtype=np.int64)
        rows = wl.store_rows(self.w, torch.as_tensor(ids), self.device)
        f32 = self.w.key_dtype == "f32"
        pre = _bits(rows["prefix"], f32)
        tok = rows["ids"].cpu().numpy()
        where = {int(j): i for i, j in enumerate(ids)}
        return oracle.decide(self.kc, self.oq["prefix"], self.oq["ids"], self.p,
                             lambda js: pre[[where[int(j)] for j in js]],
                             lambda js: tok[[where[int(j)] for j in js]])

    def pair_scores(self, b, j):
        row = wl.store_rows(self.w, torch.as_tensor([j]), self.device)
        f32 = self.w.key_dtype == "f32"
        kc = oracle.KeyCheck(self.oq["emb"][b:b + 1], -np.inf)
        kc.add_rows(_bits(row["key"], f32), j)
        r, m = oracle.lookahead(self.oq["prefix"][b], self.oq["ids"][b], _bits(row["prefix"], f32),
                                row["ids"].cpu().numpy())
        return float(kc.best[0]), float(r[0]), int(m[0]), self.w.k


def stratified_sample(classes, per_class: int, seed: int = 0):
    """Query rows to check: up to per_class of each generator class, chosen by a seeded permutation."""
    rng = np.random.default_rng(seed)
    cls = np.asarray(classes)
    rows = []
    for c in np.unique(cls):
        idx = np.nonzero(cls == c)[0]
        rows.extend(rng.permutation(idx)[:per_class].tolist())
    return np.sort(np.array(rows, dtype=np.int64))
