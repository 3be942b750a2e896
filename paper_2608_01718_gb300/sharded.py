"""Entry-range sharding of the lookup over torch.distributed ranks, one GPU each.

Rank g's handle holds the global entries [base_g, base_g + n_g), with bases increasing with the rank. A sharded
lookup of a batch runs in three steps. First each rank runs its own lookup with the candidate outputs, writing
them into a send record. Then one all-gather brings every rank's record to every rank:
record_bytes(B, top_c, m) bytes per rank, 5,632 at B = 32, top_c = 8. Finally the records are merged into the
result of one lookup over the whole store, with lacache_merge_shards on the GPU. The merge is exact: see
include/lacache.h.

The record of one rank is one uint8 buffer of typed fields. Each field is 16-byte aligned, so that rank slices of
the gathered buffer keep the alignment the kernels need:
    cand_id int32 [B, c]   cand_score F [B, c]   cand_prefix_score F [B, c]   cand_matches int32 [B, c]
    cand_prefix_scores F [B, c, m]   key_score F [B]   n_cand int32 [B]   cand_pass uint8 [B, c]
F is float32 for the GPU path. The callables that fill and merge records are the caller's, so the same exchange
carries float64 records in host-only tests.
"""
from __future__ import annotations

import torch
import torch.distributed as dist

_FIELDS = (("cand_id", torch.int32, "c"), ("cand_score", None, "c"), ("cand_prefix_score", None, "c"),
           ("cand_matches", torch.int32, "c"), ("cand_prefix_scores", None, "cm"), ("key_score", None, ""),
           ("n_cand", torch.int32, ""), ("cand_pass", torch.uint8, "c"))


def layout(B: int, top_c: int, models: int, float_dtype=torch.float32):
    """[(name, dtype, shape, byte offset)] of a record, and its size in bytes (a multiple of 16)."""
    shapes = {"c": (B, top_c), "cm": (B, top_c, models), "": (B,)}
    out, off = [], 0
    for name, dtype, kind in _FIELDS:
        dtype = dtype or float_dtype
        shape = shapes[kind]
        n = 1
        for s in shape:
            n *= s
        out.append((name, dtype, shape, off))
        off += (n * torch.empty((), dtype=dtype).element_size() + 15) // 16 * 16
    return out, off


def record_bytes(B: int, top_c: int, models: int, float_dtype=torch.float32) -> int:
    return layout(B, top_c, models, float_dtype)[1]


def views(buf: torch.Tensor, B: int, top_c: int, models: int, float_dtype=torch.float32) -> dict:
    """Typed views of the fields of one record held in the uint8 tensor buf."""
    fields, size = layout(B, top_c, models, float_dtype)
    if buf.dtype != torch.uint8 or buf.numel() != size or not buf.is_contiguous():
        raise ValueError(f"a record is a contiguous uint8 tensor of {size} bytes")
    out = {}
    for name, dtype, shape, off in fields:
        n = 1
        for s in shape:
            n *= s
        nbytes = n * torch.empty((), dtype=dtype).element_size()
        out[name] = buf[off:off + nbytes].view(dtype).view(shape)
    return out


class ShardedLookup:
    """The sharded lookup of one rank (see the module docstring).

    local_lookup(queries, record): the rank's own lookup, writing its candidate outputs into the record's views.
    merge(shards, out): merges [(record views, base)] of every rank into ``out``, the whole-store result.
    """

    def __init__(self, B: int, top_c: int, models: int, base: int, device, local_lookup, merge, group=None,
                 float_dtype=torch.float32):
        self.B, self.top_c, self.models = B, top_c, models
        self.group = group
        # without a process group: one shard, merged with itself (no exchange)
        self.world = dist.get_world_size(group) if dist.is_initialized() else 1
        self.local_lookup, self.merge = local_lookup, merge
        self.device = torch.device(device)
        size = record_bytes(B, top_c, models, float_dtype)
        # every rank's base, once: the merge needs them in rank order
        mine = torch.tensor([base], dtype=torch.int64, device=self.device)
        bases = [torch.empty_like(mine) for _ in range(self.world)]
        if self.world > 1:
            dist.all_gather(bases, mine, group=group)
        else:
            bases = [mine]
        self.bases = [int(b.item()) for b in bases]
        if any(b1 < b0 for b0, b1 in zip(self.bases, self.bases[1:])):
            raise ValueError(f"shard bases must increase with the rank: {self.bases}")
        self.send = torch.zeros(size, dtype=torch.uint8, device=self.device)
        self.gathered = (torch.zeros((self.world, size), dtype=torch.uint8, device=self.device) if self.world > 1
                         else self.send.view(1, size))
        self.local = views(self.send, B, top_c, models, float_dtype)
        self.shards = [(views(self.gathered[g], B, top_c, models, float_dtype), self.bases[g])
                       for g in range(self.world)]
        self._nccl = self.world > 1 and dist.get_backend(group) == "nccl"

    def __call__(self, queries, out):
        """Whole-store lookup of ``queries`` into ``out`` on this rank (every rank gets the same result)."""
        self.local_lookup(queries, self.local)
        if self.world == 1:
            pass
        elif self._nccl:
            dist.all_gather_into_tensor(self.gathered, self.send, group=self.group)
        else:
            dist.all_gather(list(self.gathered.unbind(0)), self.send, group=self.group)
        self.merge(self.shards, out)
        return out
