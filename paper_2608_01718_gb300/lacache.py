"""Python binding of liblacache.so (include/lacache.h): the same entry points under the same names.

Argument marshalling only. Tensors are passed by their data pointers; ``cuda_stream`` defaults to torch's current
stream on the handle's device. Every step of the lookup runs in the library's CUDA kernels. There is no CPU path:
if the library has not been built, loading it raises.
"""
from __future__ import annotations

import ctypes
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "liblacache.so")

LACACHE_OK, LACACHE_ERR_INVALID_ARG, LACACHE_ERR_CAPACITY, LACACHE_ERR_OOM = 0, 1, 2, 3
LACACHE_ERR_CUDA, LACACHE_ERR_DEVICE_TIMEOUT, LACACHE_ERR_UNSUPPORTED, LACACHE_ERR_IO = 4, 5, 6, 7
LACACHE_CHECK_EMB, LACACHE_CHECK_TOKENS, LACACHE_CHECK_BOTH = 0, 1, 2
LACACHE_BF16, LACACHE_F32 = 0, 1
LACACHE_STAGE1_AUTO, LACACHE_STAGE1_TENSOR, LACACHE_STAGE1_STREAM, LACACHE_STAGE1_LSH = 0, 1, 2, 3
LACACHE_STAGE1_TENSOR_PAIR = 4   # reported by lacache_last_launch only
LACACHE_STAGE1_LSH_TENSOR = 5    # reported by lacache_last_launch only
LACACHE_MISS_KEY, LACACHE_HIT, LACACHE_REJECT = 0, 1, 2

LACACHE_MAX_MODELS = 8
LACACHE_MAX_SHARDS = 16

EXPORTS = ["lacache_create", "lacache_create_ensemble", "lacache_destroy", "lacache_insert", "lacache_lookup",
           "lacache_lookup_host", "lacache_lookup_host_async", "lacache_append_misses", "lacache_read_rows",
           "lacache_size", "lacache_sync", "lacache_last_launch", "lacache_stage_timing", "lacache_stage_times",
           "lacache_inject_stall", "lacache_enable_lsh", "lacache_read_signatures", "lacache_calibrate",
           "lacache_calibrate_workspace_bytes", "lacache_verify_draft", "lacache_lookup_noalloc",
           "lacache_merge_shards", "lacache_get_stats", "lacache_save", "lacache_load", "lacache_get_config",
           "lacache_status_string"]


class lacache_config(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("k", ctypes.c_int32), ("capacity", ctypes.c_int64),
                ("tau_c", ctypes.c_float), ("tau_a", ctypes.c_float), ("top_c", ctypes.c_int32),
                ("token_match_min", ctypes.c_int32), ("check_mode", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("device", ctypes.c_int32), ("stage1", ctypes.c_int32)]


class lacache_ensemble(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int32), ("dims", ctypes.c_int32 * LACACHE_MAX_MODELS),
                ("tau_a", ctypes.c_float * LACACHE_MAX_MODELS)]


class lacache_result(ctypes.Structure):
    _fields_ = [(name, ctypes.c_void_p) for name in
                ("entry_id", "status", "key_score", "prefix_score", "token_matches", "n_cand",
                 "cand_id", "cand_score", "cand_prefix_score", "cand_matches", "prefix_scores", "cand_pass",
                 "cand_prefix_scores")]


class lacache_stats(ctypes.Structure):
    _fields_ = [(name, ctypes.c_int64) for name in
                ("lookups", "queries", "hits", "rejects", "key_misses", "inserted", "appended")]


class lacache_shard_result(ctypes.Structure):
    _fields_ = [(name, ctypes.c_void_p) for name in
                ("cand_id", "cand_score", "cand_prefix_score", "cand_matches", "cand_pass", "cand_prefix_scores",
                 "key_score", "n_cand")] + [("id_base", ctypes.c_int64)]


class LacacheError(RuntimeError):
    def __init__(self, call: str, status: int):
        super().__init__(f"{call}: {status_string(status)} ({status})")
        self.status = status


_lib = None


def load() -> ctypes.CDLL:
    """Open liblacache.so (once). Raises if it has not been built: there is no fallback."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2608_01718_gb300.build` "
                           "(or __graft_entry__.build()); the lookup has no CPU fallback")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    p64 = ctypes.POINTER(ctypes.c_int64)
    p32 = ctypes.POINTER(ctypes.c_int32)
    sig = {
        "lacache_create": ([ctypes.POINTER(lacache_config), ctypes.POINTER(vp)], i32),
        "lacache_create_ensemble": ([ctypes.POINTER(lacache_config), ctypes.POINTER(lacache_ensemble),
                                     ctypes.POINTER(vp)], i32),
        "lacache_destroy": ([vp], i32),
        "lacache_insert": ([vp, i64, vp, vp, vp, i32, p64, vp], i32),
        "lacache_lookup": ([vp, i32, vp, vp, vp, ctypes.POINTER(lacache_result), vp], i32),
        "lacache_lookup_host": ([vp, i32, vp, vp, vp, ctypes.POINTER(lacache_result), vp], i32),
        "lacache_lookup_host_async": ([vp, i32, vp, vp, vp, ctypes.POINTER(lacache_result), vp], i32),
        "lacache_append_misses": ([vp, i32, vp, vp, vp, vp, p64, p64, vp], i32),
        "lacache_read_rows": ([vp, i64, i64, vp, vp, vp, vp], i32),
        "lacache_size": ([vp, p64], i32),
        "lacache_sync": ([vp], i32),
        "lacache_last_launch": ([vp, p32, p32], i32),
        "lacache_stage_timing": ([vp, i32], i32),
        "lacache_stage_times": ([vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double), p64], i32),
        "lacache_inject_stall": ([vp, i32], i32),
        "lacache_enable_lsh": ([vp, i32, i32, vp, vp], i32),
        "lacache_read_signatures": ([vp, i64, i64, vp, vp], i32),
        "lacache_calibrate": ([i64, i32, vp, vp, ctypes.c_double, ctypes.c_float, vp, vp, vp, vp], i32),
        "lacache_calibrate_workspace_bytes": ([], ctypes.c_size_t),
        "lacache_verify_draft": ([i32, i32, vp, vp, vp, vp, vp], i32),
        "lacache_lookup_noalloc": ([ctypes.POINTER(lacache_config), i64, vp, vp, vp, i32, vp, vp, vp,
                                    ctypes.POINTER(lacache_result), vp], i32),
        "lacache_get_stats": ([vp, ctypes.POINTER(lacache_stats), i32], i32),
        "lacache_save": ([vp, ctypes.c_char_p], i32),
        "lacache_load": ([ctypes.c_char_p, i32, i64, ctypes.POINTER(vp)], i32),
        "lacache_get_config": ([vp, ctypes.POINTER(lacache_config), ctypes.POINTER(lacache_ensemble)], i32),
        "lacache_merge_shards": ([i32, ctypes.POINTER(lacache_shard_result), i32, i32, i32,
                                  ctypes.POINTER(lacache_result), vp], i32),
        "lacache_status_string": ([i32], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().lacache_status_string(int(status)).decode()


def _check(call: str, status: int) -> None:
    if status != LACACHE_OK:
        raise LacacheError(call, status)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(cuda_stream, device: int | None = None):
    if cuda_stream is not None:
        return cuda_stream if isinstance(cuda_stream, int) else cuda_stream.cuda_stream
    import torch
    return torch.cuda.current_stream(device).cuda_stream


def make_config(d: int, k: int, capacity: int, tau_c: float, tau_a: float, top_c: int, *, max_batch: int,
                check_mode: int = LACACHE_CHECK_EMB, token_match_min: int = 0, device: int = 0,
                stage1: int = LACACHE_STAGE1_AUTO) -> lacache_config:
    return lacache_config(d, k, capacity, tau_c, tau_a, top_c, token_match_min, check_mode, max_batch, device, stage1)


def lacache_create(cfg: lacache_config) -> int:
    h = ctypes.c_void_p()
    _check("lacache_create", load().lacache_create(ctypes.byref(cfg), ctypes.byref(h)))
    return h.value


def make_ensemble(dims, taus) -> lacache_ensemble:
    ens = lacache_ensemble()
    ens.m = len(dims)
    for i, (d, t) in enumerate(zip(dims, taus)):
        ens.dims[i] = d
        ens.tau_a[i] = t
    return ens


def lacache_create_ensemble(cfg: lacache_config, ens: lacache_ensemble) -> int:
    h = ctypes.c_void_p()
    _check("lacache_create_ensemble", load().lacache_create_ensemble(ctypes.byref(cfg), ctypes.byref(ens),
                                                                     ctypes.byref(h)))
    return h.value


def lacache_destroy(h: int) -> None:
    _check("lacache_destroy", load().lacache_destroy(h))


def lacache_insert(h: int, key, prefix, ids, dtype: int = LACACHE_BF16, cuda_stream=None) -> int:
    """Append rows (device tensors [n x d], [n x d], [n x k] int32); returns the first new entry id."""
    first = ctypes.c_int64()
    n = int(ids.shape[0])
    _check("lacache_insert", load().lacache_insert(h, n, _ptr(key), _ptr(prefix), _ptr(ids), dtype,
                                                   ctypes.byref(first), _stream(cuda_stream)))
    return first.value


def _result_struct(out: dict) -> lacache_result:
    return lacache_result(*[_ptr(out.get(name)) for name, _ in lacache_result._fields_])


def lacache_lookup(h: int, q_emb, q_prefix, q_ids, out: dict, cuda_stream=None) -> None:
    """Batched lookup; ``out`` maps lacache_result field names to caller-owned device tensors."""
    res = _result_struct(out)
    _check("lacache_lookup", load().lacache_lookup(h, int(q_emb.shape[0]), _ptr(q_emb), _ptr(q_prefix),
                                                   _ptr(q_ids), ctypes.byref(res), _stream(cuda_stream)))


def lacache_get_stats(h: int, reset: bool = False) -> dict:
    """The handle's decision counters (synchronizes its device); reset zeroes them after reading."""
    st = lacache_stats()
    _check("lacache_get_stats", load().lacache_get_stats(h, ctypes.byref(st), int(reset)))
    return {name: int(getattr(st, name)) for name, _ in lacache_stats._fields_}


def lacache_save(h: int, path: str) -> None:
    """Write the cache (configuration and valid entries) to ``path``."""
    _check("lacache_save", load().lacache_save(h, os.fsencode(path)))


def lacache_load(path: str, device: int = 0, capacity: int = 0) -> int:
    """A new handle on ``device`` from a saved cache; capacity > 0 replaces the saved capacity."""
    h = ctypes.c_void_p()
    _check("lacache_load", load().lacache_load(os.fsencode(path), device, capacity, ctypes.byref(h)))
    return h.value


def lacache_get_config(h: int) -> tuple:
    """(lacache_config, lacache_ensemble) of a handle."""
    cfg, ens = lacache_config(), lacache_ensemble()
    _check("lacache_get_config", load().lacache_get_config(h, ctypes.byref(cfg), ctypes.byref(ens)))
    return cfg, ens


def lacache_merge_shards(shards: list, top_c: int, models: int, out: dict, cuda_stream=None) -> None:
    """Merge entry-range shards' lookup outputs (``shards``: one (outputs dict, id_base) per shard, outputs as
    alloc_result(candidates=True) writes them) into ``out``, the whole-store result."""
    arr = (lacache_shard_result * len(shards))()
    for g, (o, base) in enumerate(shards):
        arr[g] = lacache_shard_result(*[_ptr(o.get(name)) for name, _ in lacache_shard_result._fields_[:-1]],
                                      int(base))
    res = _result_struct(out)
    B = int(out["status"].shape[0])
    _check("lacache_merge_shards", load().lacache_merge_shards(len(shards), arr, B, top_c, models, ctypes.byref(res),
                                                               _stream(cuda_stream)))


def lacache_lookup_host(h: int, q_emb, q_prefix, q_ids, out: dict, cuda_stream=None) -> None:
    """Lookup of host-resident queries into host-resident results (synchronous)."""
    res = _result_struct(out)
    _check("lacache_lookup_host", load().lacache_lookup_host(h, int(q_emb.shape[0]), _ptr(q_emb), _ptr(q_prefix),
                                                             _ptr(q_ids), ctypes.byref(res), _stream(cuda_stream)))


def lacache_lookup_host_async(h: int, q_emb, q_prefix, q_ids, out: dict, cuda_stream=None) -> None:
    """Lookup of queries in pinned host tensors into pinned host results, enqueued on the stream without waiting:
    the results are there once the stream has passed the call."""
    res = _result_struct(out)
    _check("lacache_lookup_host_async", load().lacache_lookup_host_async(
        h, int(q_emb.shape[0]), _ptr(q_emb), _ptr(q_prefix), _ptr(q_ids), ctypes.byref(res), _stream(cuda_stream)))


def lacache_append_misses(h: int, q_emb, q_prefix, q_ids, status, cuda_stream=None) -> tuple[int, int]:
    """Append every non-HIT query of a looked-up batch in query order; returns (first id, count)."""
    first, n = ctypes.c_int64(), ctypes.c_int64()
    _check("lacache_append_misses", load().lacache_append_misses(
        h, int(q_emb.shape[0]), _ptr(q_emb), _ptr(q_prefix), _ptr(q_ids), _ptr(status), ctypes.byref(first),
        ctypes.byref(n), _stream(cuda_stream)))
    return first.value, n.value


def lacache_read_rows(h: int, first: int, n: int, key=None, prefix=None, ids=None, cuda_stream=None) -> None:
    _check("lacache_read_rows", load().lacache_read_rows(h, first, n, _ptr(key), _ptr(prefix), _ptr(ids),
                                                         _stream(cuda_stream)))


def lacache_size(h: int) -> int:
    n = ctypes.c_int64()
    _check("lacache_size", load().lacache_size(h, ctypes.byref(n)))
    return n.value


def lacache_sync(h: int) -> None:
    _check("lacache_sync", load().lacache_sync(h))


def lacache_last_launch(h: int) -> tuple[int, int]:
    splits, kernel = ctypes.c_int32(), ctypes.c_int32()
    _check("lacache_last_launch", load().lacache_last_launch(h, ctypes.byref(splits), ctypes.byref(kernel)))
    return splits.value, kernel.value


def lacache_stage_timing(h: int, max_lookups: int) -> None:
    _check("lacache_stage_timing", load().lacache_stage_timing(h, max_lookups))


def lacache_stage_times(h: int) -> tuple[float, float, int]:
    """(stage-1 ms, stage-2 ms, lookups timed) summed since the previous call."""
    t1, t2, n = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check("lacache_stage_times", load().lacache_stage_times(h, ctypes.byref(t1), ctypes.byref(t2), ctypes.byref(n)))
    return t1.value, t2.value, n.value


def lacache_inject_stall(h: int, lookups: int) -> None:
    _check("lacache_inject_stall", load().lacache_inject_stall(h, lookups))


def lacache_enable_lsh(h: int, bits: int, radius: int, hyperplanes, cuda_stream=None) -> None:
    """Build the SimHash index: signatures of every entry against hyperplanes ([bits x d] bf16)."""
    _check("lacache_enable_lsh", load().lacache_enable_lsh(h, bits, radius, _ptr(hyperplanes), _stream(cuda_stream)))


def lacache_read_signatures(h: int, first: int, n: int, out, cuda_stream=None) -> None:
    _check("lacache_read_signatures", load().lacache_read_signatures(h, first, n, _ptr(out), _stream(cuda_stream)))


def lacache_calibrate_workspace_bytes() -> int:
    return int(load().lacache_calibrate_workspace_bytes())


def lacache_calibrate(x, y, percentile: float, cap: float, sims, result, workspace, cuda_stream=None) -> None:
    """Pair similarities of (x_i, y_i) into sims, then result = [nearest-rank percentile, min(cap, it)]."""
    _check("lacache_calibrate", load().lacache_calibrate(int(x.shape[0]), int(x.shape[1]), _ptr(x), _ptr(y),
                                                         float(percentile), float(cap), _ptr(sims), _ptr(result),
                                                         _ptr(workspace), _stream(cuda_stream)))


def lacache_verify_draft(p_target, p_draft, status, accepted, cuda_stream=None) -> None:
    """Accepted draft-prefix length per query (P_f >= P_g from the first token on); -1 for served queries."""
    B, k = int(p_target.shape[0]), int(p_target.shape[1])
    _check("lacache_verify_draft", load().lacache_verify_draft(B, k, _ptr(p_target), _ptr(p_draft), _ptr(status),
                                                               _ptr(accepted), _stream(cuda_stream)))


def lacache_lookup_noalloc(cfg: lacache_config, key, prefix, ids, q_emb, q_prefix, q_ids, out: dict,
                           cuda_stream=None) -> None:
    """Lookup against caller-owned cache rows with no device allocation (see include/lacache.h)."""
    res = _result_struct(out)
    n = int(ids.shape[0]) if ids is not None else 0
    _check("lacache_lookup_noalloc", load().lacache_lookup_noalloc(
        ctypes.byref(cfg), n, _ptr(key), _ptr(prefix), _ptr(ids), int(q_emb.shape[0]), _ptr(q_emb),
        _ptr(q_prefix), _ptr(q_ids), ctypes.byref(res), _stream(cuda_stream, cfg.device)))


def alloc_result(batch: int, top_c: int, device, candidates: bool = True, pinned: bool = False,
                 models: int = 0) -> dict:
    """Output buffers of one lookup: device tensors (or pinned host tensors with ``device="cpu"``). ``candidates``
    adds the per-candidate arrays (with their pass bits); ``models`` > 0 adds every model's lookahead scores, for
    the shown candidate and, with ``candidates``, per candidate."""
    import torch
    kw = {"device": device}
    if pinned:
        kw["pin_memory"] = True
    out = {"entry_id": torch.empty(batch, dtype=torch.int32, **kw),
           "status": torch.empty(batch, dtype=torch.uint8, **kw),
           "key_score": torch.empty(batch, dtype=torch.float32, **kw),
           "prefix_score": torch.empty(batch, dtype=torch.float32, **kw),
           "token_matches": torch.empty(batch, dtype=torch.int32, **kw),
           "n_cand": torch.empty(batch, dtype=torch.int32, **kw)}
    if candidates:
        out.update({"cand_id": torch.empty((batch, top_c), dtype=torch.int32, **kw),
                    "cand_score": torch.empty((batch, top_c), dtype=torch.float32, **kw),
                    "cand_prefix_score": torch.empty((batch, top_c), dtype=torch.float32, **kw),
                    "cand_matches": torch.empty((batch, top_c), dtype=torch.int32, **kw),
                    "cand_pass": torch.empty((batch, top_c), dtype=torch.uint8, **kw)})
    if models:
        out["prefix_scores"] = torch.empty((batch, models), dtype=torch.float32, **kw)
        if candidates:
            out["cand_prefix_scores"] = torch.empty((batch, top_c, models), dtype=torch.float32, **kw)
    return out


class LaCache:
    """A handle with its configuration: thin convenience over the functions above."""

    def __init__(self, d: int, k: int, capacity: int, tau_c: float, tau_a: float, top_c: int, *, max_batch: int,
                 check_mode: int = LACACHE_CHECK_EMB, token_match_min: int = 0, device: int = 0,
                 stage1: int = LACACHE_STAGE1_AUTO, prefix_dims=None, tau_a_models=None):
        self.cfg = make_config(d, k, capacity, tau_c, tau_a, top_c, max_batch=max_batch, check_mode=check_mode,
                               token_match_min=token_match_min, device=device, stage1=stage1)
        self.device = device
        self.h = None
        if prefix_dims is None:
            self.models = 1
            self.h = lacache_create(self.cfg)
        else:
            self.models = len(prefix_dims)
            self.h = lacache_create_ensemble(self.cfg, make_ensemble(prefix_dims, tau_a_models))

    @classmethod
    def load(cls, path: str, device: int = 0, capacity: int = 0) -> "LaCache":
        """A cache saved with save(), on ``device``."""
        obj = cls.__new__(cls)
        obj.h = lacache_load(path, device, capacity)
        obj.cfg, ens = lacache_get_config(obj.h)
        obj.device = device
        obj.models = int(ens.m)
        return obj

    def save(self, path: str) -> None:
        lacache_save(self.h, path)

    def close(self) -> None:
        if self.h:
            lacache_destroy(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def insert(self, key, prefix, ids, dtype: int = LACACHE_BF16, cuda_stream=None) -> int:
        return lacache_insert(self.h, key, prefix, ids, dtype, cuda_stream)

    def lookup(self, q_emb, q_prefix, q_ids, out: dict | None = None, candidates: bool = True,
               cuda_stream=None) -> dict:
        if out is None:
            out = alloc_result(q_emb.shape[0], self.cfg.top_c, q_emb.device, candidates, models=self.models)
        lacache_lookup(self.h, q_emb, q_prefix, q_ids, out, cuda_stream)
        return out

    def stats(self, reset: bool = False) -> dict:
        return lacache_get_stats(self.h, reset)

    def append_misses(self, q_emb, q_prefix, q_ids, status, cuda_stream=None) -> tuple[int, int]:
        return lacache_append_misses(self.h, q_emb, q_prefix, q_ids, status, cuda_stream)

    @property
    def size(self) -> int:
        return lacache_size(self.h)

    def sync(self) -> None:
        lacache_sync(self.h)

    def last_launch(self) -> tuple[int, int]:
        return lacache_last_launch(self.h)
