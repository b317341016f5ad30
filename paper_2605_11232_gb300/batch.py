"""Set up a workload's KV cache through the C ABI and hold its device buffers.

This is the harness a serving engine would be: it allocates the pool and the
caches (torch device memory), pins each shared prefix in refcounted blocks,
gives every request its block-table row (prefix blocks retained, private
blocks allocated), and writes the cached tokens with ``kv_cache_write``.  The
step's own inputs (new-token K/V, queries, slot mapping) are staged on the
device so a benchmark step reads them from HBM.  All arithmetic of the path
happens in the library's kernels.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

from . import pkv
from .workloads import Workload


def _blocks(n: int) -> int:
    return (int(n) + 15) // 16


@dataclass
class Batch:
    w: Workload
    device: torch.device
    pool: object
    k_cache: torch.Tensor
    v_cache: torch.Tensor
    table_host: np.ndarray          # [R][max_blocks] int32, -1 padded
    prefix_ids: list                # per group: int32 ids
    slots_host: np.ndarray          # [T] slots of this step's new tokens
    # device copies
    table: torch.Tensor
    context_lens: torch.Tensor
    slots: torch.Tensor
    k_new: torch.Tensor
    v_new: torch.Tensor
    q: torch.Tensor
    # decode subset (contiguous request range) and prefill subset
    dec: slice
    pre: slice
    cu_pre: torch.Tensor            # [Rp+1] cu_seqlens of the prefill subset
    max_seqlen_pre: int
    groups_dev: dict                # device arrays of the decode prefix groups
    groups: object                  # pkv.PrefixGroups for the decode subset (or None)
    num_blocks_pool: int = 0

    def close(self):
        if self.pool is not None:
            pkv.kv_pool_destroy(self.pool)
            self.pool = None


def _contiguous_range(idx: np.ndarray) -> slice:
    if len(idx) == 0:
        return slice(0, 0)
    assert np.array_equal(idx, np.arange(idx[0], idx[-1] + 1)), "subset must be contiguous"
    return slice(int(idx[0]), int(idx[-1]) + 1)


def build_batch(w: Workload, device="cuda", poison: bool = True, placement_seed=None,
                share_prefix: bool = True, table_width: int | None = None) -> Batch:
    """Allocate the pool, write every cached token, stage this step's inputs.

    poison: fill the caches with bf16 NaN first, so any read of a slot that
    holds no token shows up in the outputs.
    share_prefix: False gives every request a private copy of its group's
    prefix (the "no APC" layout), used to check shared == private.
    """
    dev = torch.device(device)
    nb = w.num_blocks
    if not share_prefix:
        nb = w.num_blocks + sum(_blocks(w.prefix_len_of(r)) for r in range(w.num_requests))
    shape = (nb, w.num_kv_heads, 16, w.head_dim)
    if poison:
        k_cache = torch.full(shape, float("nan"), dtype=torch.bfloat16, device=dev)
        v_cache = torch.full(shape, float("nan"), dtype=torch.bfloat16, device=dev)
    else:
        k_cache = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
        v_cache = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    seed = w.placement_seed if placement_seed is None else placement_seed
    pool = pkv.kv_pool_create(nb, w.num_kv_heads, w.head_dim, k_cache, v_cache,
                              placement_seed=seed)
    R = w.num_requests
    ctx = w.context_lens
    nblk = np.array([_blocks(c) for c in ctx], np.int64)
    width = int(nblk.max()) if table_width is None else int(table_width)
    table = np.full((R, width), -1, np.int32)

    def write(k_rows: torch.Tensor, v_rows: torch.Tensor, slots: np.ndarray):
        if len(slots) == 0:
            return
        kd = k_rows.to(dev, non_blocking=False).contiguous()
        vd = v_rows.to(dev, non_blocking=False).contiguous()
        sd = torch.from_numpy(np.ascontiguousarray(slots, np.int64)).to(dev)
        pkv.kv_cache_write(pool, kd, vd, sd)

    # shared prefixes: allocated once, refcount 1 held by the prefix registry
    prefix_ids = []
    for g, P in enumerate(w.prefix_lens):
        ids = pkv.kv_pool_alloc(pool, _blocks(P))
        prefix_ids.append(ids)
        if share_prefix:
            slots = pkv.kv_slot_mapping(pool, ids[None, :], [P], [P])
            write(w.prefix_k[g], w.prefix_v[g], slots)
    # per request: table row = retained prefix blocks + private blocks
    for r in range(R):
        g = int(w.group_of_req[r])
        P = w.prefix_len_of(r)
        if share_prefix and g >= 0:
            row = pkv.kv_pool_alloc_sequence(pool, prefix_ids[g], int(nblk[r]))
        else:
            row = pkv.kv_pool_alloc_sequence(pool, None, int(nblk[r]))
        table[r, : nblk[r]] = row
    # cached tokens not covered by a shared prefix
    for r in range(R):
        g = int(w.group_of_req[r])
        P = w.prefix_len_of(r) if share_prefix else 0
        cached = int(w.cached_lens[r])
        if cached <= P:
            continue
        n_priv_cached = cached - P
        slots = pkv.kv_slot_mapping(pool, table[r:r + 1], [cached], [n_priv_cached])
        a, b = int(w.priv_off[r]), int(w.priv_off[r + 1])
        if share_prefix or g < 0:
            write(w.priv_k[a:b], w.priv_v[a:b], slots)
        else:   # private copy: the prefix tokens first, then the request's own
            Pg = w.prefix_len_of(r)
            write(torch.cat([w.prefix_k[g], w.priv_k[a:b]]),
                  torch.cat([w.prefix_v[g], w.priv_v[a:b]]), slots)
    torch.cuda.synchronize(dev)
    # this step's new tokens
    slots_host = pkv.kv_slot_mapping(pool, table, ctx, w.new_lens)
    dec = _contiguous_range(w.subset(True))
    pre = _contiguous_range(w.subset(False))
    cu_pre_h = np.zeros(pre.stop - pre.start + 1, np.int32)
    cu_pre_h[1:] = np.cumsum(w.new_lens[pre])
    groups_dev, groups = {}, None
    Rd = dec.stop - dec.start
    if share_prefix and Rd > 0:
        gor = w.group_of_req[dec].astype(np.int32)
        G = len(w.prefix_lens)
        members = [np.nonzero(gor == g)[0].astype(np.int32) for g in range(G)]
        gstart = np.zeros(G + 1, np.int32)
        gstart[1:] = np.cumsum([len(m) for m in members])
        gblocks = np.array([P // 16 for P in w.prefix_lens], np.int32)
        groups_dev = dict(
            group_start=torch.from_numpy(gstart).to(dev),
            member_req=torch.from_numpy(np.concatenate(members) if G else np.zeros(0, np.int32)).to(dev),
            group_blocks=torch.from_numpy(gblocks).to(dev),
            group_of_req=torch.from_numpy(gor).to(dev),
        )
        groups = pkv.make_prefix_groups(G, int(gblocks.max()) if G else 0,
                                        max(len(m) for m in members) if G else 0, **groups_dev)
    b = Batch(
        w=w, device=dev, pool=pool, k_cache=k_cache, v_cache=v_cache, table_host=table,
        prefix_ids=prefix_ids, slots_host=slots_host,
        table=torch.from_numpy(table).to(dev),
        context_lens=torch.from_numpy(ctx.astype(np.int32)).to(dev),
        slots=torch.from_numpy(slots_host).to(dev),
        k_new=w.new_k.to(dev), v_new=w.new_v.to(dev), q=w.q.to(dev),
        dec=dec, pre=pre, cu_pre=torch.from_numpy(cu_pre_h).to(dev),
        max_seqlen_pre=int(w.new_lens[pre].max()) if pre.stop > pre.start else 0,
        groups_dev=groups_dev, groups=groups, num_blocks_pool=nb)
    return b


def step_view(buf: torch.Tensor, off: int, like: torch.Tensor) -> torch.Tensor:
    """The region of a packed uint8 step buffer at byte offset `off`, viewed
    with the dtype and shape of `like`."""
    nb = like.numel() * like.element_size()
    return buf[off:off + nb].view(like.dtype).view(like.shape)


def step_buffers(b: Batch, copies: int = 2, fused: bool = False):
    """Packed inputs of one decode step of a decode-only batch (q, new K/V,
    slot mapping, context lengths; 256-byte aligned regions): the
    pkv.StepLayout, `copies` pinned host buffers holding them, and a device
    buffer of the same size.  fused: the decode kernels store the new K/V
    (PKV_STEP_FUSED_WRITE), and the packed buffer holds no slot mapping."""
    if b.pre.stop != b.pre.start:
        raise ValueError("step buffers are for decode-only batches")
    parts = [pt for pt in step_parts(b) if not (fused and pt[0] == "slot_mapping")]
    offs, n = {}, 0
    for name, t in parts:
        offs[name] = n
        n += (t.numel() * t.element_size() + 255) // 256 * 256
    layout = pkv.StepLayout(bytes=n, flags=pkv.PKV_STEP_FUSED_WRITE if fused else 0, **offs)
    hosts = [torch.empty(n, dtype=torch.uint8).pin_memory() for _ in range(copies)]
    for h in hosts:
        for name, t in parts:
            step_view(h, offs[name], t).copy_(t.cpu())
    dev = torch.empty(n, dtype=torch.uint8, device=b.device)
    return layout, hosts, dev


def step_parts(b: Batch):
    """(field of pkv.StepLayout, device tensor) of a batch's step inputs."""
    return [("q", b.q), ("k_new", b.k_new), ("v_new", b.v_new), ("slot_mapping", b.slots),
            ("context_lens", b.context_lens)]


def new_token_rows(w: Workload, req: slice) -> slice:
    """Rows of q / k_new belonging to a contiguous request range."""
    return slice(int(w.cu_new[req.start]), int(w.cu_new[req.stop]))


def run_write(b: Batch, stream=None):
    pkv.kv_cache_write(b.pool, b.k_new, b.v_new, b.slots, stream)


def decode_workspace(b: Batch, use_groups: bool = True) -> torch.Tensor:
    Rd = b.dec.stop - b.dec.start
    nbytes = pkv.paged_attn_decode_workspace_size(
        b.pool, Rd, b.w.num_q_heads, b.table.shape[1], b.groups if use_groups else None)
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=b.device)


def run_decode(b: Batch, out: torch.Tensor, lse, ws: torch.Tensor, use_groups: bool = True,
               stream=None):
    rows = new_token_rows(b.w, b.dec)
    pkv.paged_attn_decode(b.pool, b.q[rows], out, lse, b.context_lens[b.dec], b.table[b.dec],
                          b.w.scale, b.groups if use_groups else None, ws, stream)


def run_decode_append(b: Batch, out: torch.Tensor, lse, ws: torch.Tensor, use_groups: bool = True,
                      stream=None):
    """The decode subset's cache write and attention in one call: each decode
    request's new K/V row is stored by the decode kernels."""
    rows = new_token_rows(b.w, b.dec)
    pkv.paged_attn_decode_append(b.pool, b.q[rows], b.k_new[rows], b.v_new[rows], out, lse,
                                 b.context_lens[b.dec], b.table[b.dec], b.w.scale,
                                 b.groups if use_groups else None, ws, stream)


def run_prefill(b: Batch, out: torch.Tensor, lse, stream=None):
    rows = new_token_rows(b.w, b.pre)
    pkv.paged_attn_prefill(b.pool, b.q[rows], out, lse, b.cu_pre, b.context_lens[b.pre],
                           b.table[b.pre], b.max_seqlen_pre, b.w.scale, stream)


def run_prefill_append(b: Batch, out: torch.Tensor, lse, stream=None):
    """The prefill subset's cache write and attention in one call: the
    prefill kernel stores each new token's K/V."""
    rows = new_token_rows(b.w, b.pre)
    pkv.paged_attn_prefill_append(b.pool, b.q[rows], b.k_new[rows], b.v_new[rows], out, lse, b.cu_pre,
                                  b.context_lens[b.pre], b.table[b.pre], b.max_seqlen_pre, b.w.scale, stream)


def verify_groups(b: Batch):
    """Token groups of the prefill subset's requests for grouped verification:
    (pkv.VerifyGroups, the device tensors it points to; keep them alive)."""
    w = b.w
    req = range(b.pre.start, b.pre.stop)
    G = len(w.prefix_lens)
    rg = np.array([int(w.group_of_req[r]) for r in req], np.int32)
    cu = np.zeros(len(rg) + 1, np.int32)
    cu[1:] = np.cumsum(w.new_lens[b.pre])
    tg = pkv.pkv_verify_groups_build(cu, rg, G)
    gblocks = np.array([P // 16 for P in w.prefix_lens], np.int32)
    dev = dict(group_start=torch.from_numpy(tg["group_start"]).to(b.device),
               member_token=torch.from_numpy(tg["member_token"]).to(b.device),
               group_blocks=torch.from_numpy(gblocks).to(b.device),
               group_row=torch.from_numpy(tg["group_row"]).to(b.device),
               request_group=torch.from_numpy(rg).to(b.device))
    vg = pkv.make_verify_groups(G, int(gblocks.max()) if G else 0, tg["max_group_tokens"], **dev)
    return vg, dev


def verify_workspace(b: Batch, groups) -> torch.Tensor:
    rows = new_token_rows(b.w, b.pre)
    nbytes = pkv.paged_attn_verify_tree_workspace_size(b.pool, rows.stop - rows.start, b.w.num_q_heads,
                                                       b.table.shape[1], groups)
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=b.device)


def run_verify_grouped(b: Batch, out: torch.Tensor, lse, tree_mask: torch.Tensor, groups, ws: torch.Tensor,
                       max_seqlen_q: int | None = None, stream=None):
    rows = new_token_rows(b.w, b.pre)
    pkv.paged_attn_verify_tree_grouped(b.pool, b.q[rows], out, lse, b.cu_pre, b.context_lens[b.pre],
                                       b.table[b.pre], max_seqlen_q or b.max_seqlen_pre, b.w.scale, tree_mask,
                                       groups, ws, stream)


def kv_waste(b: Batch) -> float:
    """Fraction of allocated KV slots holding no token, shared blocks once."""
    used_blocks = b.num_blocks_pool - pkv.kv_pool_num_free(b.pool)
    tokens = sum(b.w.prefix_lens) + sum(
        int(b.w.context_lens[r]) - b.w.prefix_len_of(r) for r in range(b.w.num_requests))
    return 1.0 - tokens / (16.0 * used_blocks)
