"""Partition of the SAKI path over several GPUs (one process per GPU).

The path shards two ways, and neither needs a collective inside a step's
arithmetic:

* By head.  Fit, index, selection and recall are independent per query head
  (Sec. 6 fits one map per head; a query head reads only its own GQA KV
  head).  Each rank owns a contiguous block of KV heads together with their
  query heads, so a GQA group never straddles two ranks; the only exchange is
  the per-head recall, gathered for the median over heads (Tab. 1 reports
  medians).
* By key range.  A long decode cache (Sec. 1's million-token setting) is split
  into contiguous key ranges, one per rank.  Each rank selects the top k of its
  range (saki_score_topk with part-local indices); one all-gather of the k
  (index, score) candidates per (head, query) brings every part to every rank,
  and saki_merge_topk keeps the k best of the union, which is the top k over
  the whole range (the ranking is a total order: descending score, then lower
  index).

Collectives go through ``torch.distributed`` (NCCL on GPUs, gloo on CPU); the
functions take the tensors a rank holds and return what the exchange gives it.
"""
from __future__ import annotations

__all__ = ["block", "head_range", "key_range", "gather_head_values", "exchange_candidates",
           "merged_topk"]


def block(n: int, world: int, rank: int) -> tuple[int, int]:
    """[lo, hi) of rank's share of n items in contiguous blocks, the first
    n % world ranks one item larger."""
    if world < 1 or not 0 <= rank < world or n < 0:
        raise ValueError("need world >= 1, 0 <= rank < world, n >= 0")
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def head_range(num_q_heads: int, num_kv_heads: int, world: int, rank: int) -> tuple[int, int, int, int]:
    """(q_lo, q_hi, kv_lo, kv_hi): the query and KV heads rank owns.  KV heads are
    split in contiguous blocks and each brings its G = Hq / Hk query heads
    (query head h reads KV head h // G)."""
    if num_kv_heads < 1 or num_q_heads % num_kv_heads:
        raise ValueError("num_q_heads must be a multiple of num_kv_heads")
    G = num_q_heads // num_kv_heads
    g0, g1 = block(num_kv_heads, world, rank)
    return g0 * G, g1 * G, g0, g1


def key_range(num_keys: int, world: int, rank: int) -> tuple[int, int]:
    """[lo, hi): rank's contiguous share of a sequence's keys."""
    return block(num_keys, world, rank)


def gather_head_values(local, num_q_heads: int, num_kv_heads: int, group=None):
    """All ranks' per-head values (e.g. recall), in global head order, on every
    rank; `local` holds this rank's heads (head_range order).  One all-gather of
    a padded tensor (shares differ by at most one GQA group)."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    G = num_q_heads // num_kv_heads
    width = -(-num_kv_heads // world) * G
    buf = torch.full((width,), float("nan"), dtype=local.dtype, device=local.device)
    buf[:local.numel()] = local
    out = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(out, buf, group=group)
    parts = []
    for r in range(world):
        q0, q1, _, _ = head_range(num_q_heads, num_kv_heads, world, r)
        parts.append(out[r][:q1 - q0])
    return torch.cat(parts)


def exchange_candidates(idx, score, key_lo: int, group=None):
    """The exchange step of a key-range split: every rank's local top-k lists
    (idx int32 with part-local indices and -1 padding, score float32, same shape
    on every rank) and range offsets, on every rank.  Returns (idx_parts,
    score_parts, offsets): tensors [world, *shape] and a list of ints."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    ib = [torch.empty_like(idx) for _ in range(world)]
    sb = [torch.empty_like(score) for _ in range(world)]
    dist.all_gather(ib, idx.contiguous(), group=group)
    dist.all_gather(sb, score.contiguous(), group=group)
    off = torch.tensor([int(key_lo)], dtype=torch.int64, device=idx.device)
    ob = [torch.empty_like(off) for _ in range(world)]
    dist.all_gather(ob, off, group=group)
    return torch.stack(ib), torch.stack(sb), [int(o.item()) for o in ob]


def merged_topk(cfg, idx_parts, score_parts, offsets, idx, score=None, stream=None):
    """saki_merge_topk on the exchanged lists (device tensors): the k best of the
    union, with global indices, into idx (and score)."""
    from . import saki
    saki.saki_merge_topk(cfg, idx_parts, score_parts, offsets, idx, score=score, stream=stream)
