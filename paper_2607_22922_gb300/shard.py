"""Row-sharded search: one index split by rows over G processes, one GPU each.

The paper runs on one device; its three stages (§2: Filter, Rank, Select)
are per row up to the final Select, so an index splits by rows without
changing any result.  Process g holds rows [r_g, r_{g+1}) (codes and
attribute columns), runs Filter, Rank and the per-shard Select on them with
its own library index, and turns its local row ids into global ones by
adding r_g.  One exchange follows: every process gathers the G per-shard
lists of k (dist, id) per query (an all-gather of nq * k * 12 bytes per
shard) and the pass counts (a sum), and ``ifvs_merge_topk`` keeps the k
smallest by (dist, id).  A shard's k best contain every row of the global
k best that lies in the shard, and local id order is global id order
inside a shard, so the merged lists equal one search over all rows.

The collective is torch.distributed's (NCCL on GPUs, gloo on CPU); the
merge is the library's kernel.  Queries, predicates and w_z are the same on
every process.
"""
from __future__ import annotations

import numpy as np


def shard_bounds(N: int, world: int, rank: int, align: int = 1024) -> tuple:
    """Rows [r0, r1) of shard ``rank`` of ``world``: contiguous, in rank
    order, sizes multiples of ``align`` rows except the last shard's."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank %d outside 0..%d" % (rank, world - 1))
    blocks = (N + align - 1) // align
    per = blocks // world
    extra = blocks % world
    b0 = rank * per + min(rank, extra)
    b1 = b0 + per + (1 if rank < extra else 0)
    return min(N, b0 * align), min(N, b1 * align)


def offset_ids(ids, r0: int):
    """Local row ids -> global ones (-1 padding kept); torch tensor or numpy."""
    if isinstance(ids, np.ndarray):
        return np.where(ids >= 0, ids + r0, ids)
    import torch
    return torch.where(ids >= 0, ids + r0, ids)


def gather_results(dists, ids, npass, group=None):
    """All-gather of every shard's [nq][k] dists and global ids (torch
    tensors on the collective's device) into [G][nq][k] tensors, in rank
    order, and the sum of the per-shard pass counts [nq]."""
    import torch
    import torch.distributed as dist
    G = dist.get_world_size(group)
    dl = [torch.empty_like(dists) for _ in range(G)]
    il = [torch.empty_like(ids) for _ in range(G)]
    dist.all_gather(dl, dists.contiguous(), group=group)
    dist.all_gather(il, ids.contiguous(), group=group)
    total = npass.clone()
    dist.all_reduce(total, op=dist.ReduceOp.SUM, group=group)
    return torch.stack(dl), torch.stack(il), total


class ShardedIndex:
    """This process's shard of a row-sharded index (rows [r0, r1) of the
    whole), on ``device``; ``search`` returns the results over all shards."""

    def __init__(self, codes, attrs, r0: int, device: int = 0, group=None, **kw):
        from paper_2607_22922_gb300 import ifvs
        self.ifvs = ifvs
        self.r0 = int(r0)
        self.device = device
        self.group = group
        self.local = ifvs.Index(codes, attrs, device=device, **kw)

    def load_codebooks(self, *a, **kw):
        self.local.load_codebooks(*a, **kw)
        return self

    def search(self, queries, preds, k, wz, stream=None, **kw):
        """queries [nq][D] float32, preds (104-byte records, as uint8
        [nq][104]) and wz [nq][D] as device tensors; returns device tensors
        ids [nq][k] (global rows), dists [nq][k], npass [nq] (all shards)."""
        import torch
        ifvs = self.ifvs
        nq = int(queries.shape[0])
        dev = queries.device
        ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
        d = torch.empty((nq, k), dtype=torch.float32, device=dev)
        npass = torch.empty(nq, dtype=torch.int64, device=dev)
        # the library runs on torch's stream, after the work that produced the inputs
        stream = stream if stream is not None else torch.cuda.current_stream(dev)
        sptr = stream.cuda_stream
        ifvs.ifvs_search_batch(self.local.h, queries, preds, k, wz=wz, ids=ids, dists=d, npass=npass,
                               flags=ifvs.IFVS_F_DEVICE_IO, stream=sptr, **kw)
        stream.synchronize()
        ids = offset_ids(ids, self.r0)
        all_d, all_i, total = gather_results(d, ids, npass, self.group)
        out_i = torch.empty((nq, k), dtype=torch.int64, device=dev)
        out_d = torch.empty((nq, k), dtype=torch.float32, device=dev)
        ifvs.ifvs_merge_topk(all_d, all_i, k, device=self.device, dists_out=out_d, ids_out=out_i,
                             flags=ifvs.IFVS_F_DEVICE_IO, stream=sptr)
        stream.synchronize()
        return out_i, out_d, total

    def close(self):
        self.local.close()
