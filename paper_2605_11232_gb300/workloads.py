"""Seeded synthetic workloads for prefix-cached paged attention.

This module only decides *shapes and values*: how many requests, which shared
prefix each one uses, how many tokens are already cached, how many are new, and
the bf16 query/key/value numbers drawn from N(0, 1).  It contains none of the
attention arithmetic, no block allocation and no block-table construction, so
both the CUDA path and the fp64 oracle can consume it without sharing any
method code.

The five workloads restate the paper's serving scenarios as attention shapes:
a long reusable policy/schema prefix shared by many requests (Sec. 5.4, prefix
reuse and KV management), short case-specific suffixes, short structured outputs
(Sec. 5.3, 50-75 generated tokens) and a multi-tenant mix of prefixes (Sec. 3,
workload characterisation; Table "phenotype").  The paper's own inputs (IBM AML
and SAML-D rendered into prompts, Table "publicdata") are replaced by random
tensors of the same lengths: attention cost and numerics depend only on shapes.

Draw order (fixed, so a seed names one workload): lengths -> placement seed ->
prefix K/V per group -> cached private K/V per request -> new-token K/V -> Q.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

BLOCK_SIZE = 16
BASE_SEED = 20260

# name -> index (the seed of workload i is BASE_SEED + i)
WORKLOAD_NAMES = ["tiny", "l8b_decode", "l8b_prefill", "qwen_mixed", "l70b_decode"]


@dataclass
class Workload:
    """One batch of requests over a paged KV cache with shared prefixes.

    Per request r (index order = the order of rows in ``q``/``k_new``):
      group_of_req[r]  shared-prefix group (-1: none); the group's prefix is
                       the first prefix_lens[g] tokens of the request
      cached_lens[r]   tokens already in the KV cache before this step
                       (prefix + private cached tokens)
      new_lens[r]      tokens produced this step (1 = decode query)
      is_decode[r]     True for decode requests, False for prefill/chunk
    Context length L_r = cached_lens[r] + new_lens[r].  New token i of request
    r sits at absolute position cached_lens[r] + i.
    """

    name: str
    seed: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    block_size: int
    prefix_lens: list
    group_of_req: np.ndarray
    cached_lens: np.ndarray
    new_lens: np.ndarray
    is_decode: np.ndarray
    num_blocks: int
    placement_seed: int
    # values, all bf16 CPU tensors
    prefix_k: list = field(default_factory=list)   # [P_g][Hkv][d]
    prefix_v: list = field(default_factory=list)
    priv_k: torch.Tensor = None                    # [sum private cached][Hkv][d]
    priv_v: torch.Tensor = None
    priv_off: np.ndarray = None                    # [R+1] offsets into priv_k
    new_k: torch.Tensor = None                     # [T][Hkv][d]
    new_v: torch.Tensor = None
    q: torch.Tensor = None                         # [T][Hq][d]
    cu_new: np.ndarray = None                      # [R+1] offsets into new_k / q

    @property
    def num_requests(self) -> int:
        return int(self.cached_lens.shape[0])

    @property
    def context_lens(self) -> np.ndarray:
        return (self.cached_lens + self.new_lens).astype(np.int32)

    @property
    def num_new_tokens(self) -> int:
        return int(self.cu_new[-1])

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.head_dim)

    def prefix_len_of(self, r: int) -> int:
        g = int(self.group_of_req[r])
        return 0 if g < 0 else int(self.prefix_lens[g])

    def request_kv(self, r: int):
        """Logical K and V of request r, contiguous [L_r][Hkv][d] bf16 (prefix,
        cached private tokens, new tokens, in position order)."""
        parts_k, parts_v = [], []
        g = int(self.group_of_req[r])
        if g >= 0:
            parts_k.append(self.prefix_k[g])
            parts_v.append(self.prefix_v[g])
        a, b = int(self.priv_off[r]), int(self.priv_off[r + 1])
        parts_k.append(self.priv_k[a:b])
        parts_v.append(self.priv_v[a:b])
        a, b = int(self.cu_new[r]), int(self.cu_new[r + 1])
        parts_k.append(self.new_k[a:b])
        parts_v.append(self.new_v[a:b])
        return torch.cat(parts_k, 0), torch.cat(parts_v, 0)

    def request_q(self, r: int) -> torch.Tensor:
        a, b = int(self.cu_new[r]), int(self.cu_new[r + 1])
        return self.q[a:b]

    def subset(self, decode: bool):
        """Indices of the decode (or the prefill) requests."""
        return np.nonzero(self.is_decode == decode)[0]


def _randn_bf16(gen: torch.Generator, shape) -> torch.Tensor:
    """N(0, 1) fp32 draws rounded to bf16 (round-to-nearest-even)."""
    n = int(np.prod(shape))
    if n == 0:
        return torch.empty(shape, dtype=torch.bfloat16)
    return torch.randn(shape, generator=gen, dtype=torch.float32).to(torch.bfloat16)


def _uniform_int(gen: torch.Generator, lo: int, hi: int, n: int) -> np.ndarray:
    """n integers uniform on [lo, hi] inclusive."""
    return torch.randint(lo, hi + 1, (n,), generator=gen).numpy().astype(np.int64)


def _log_uniform_int(gen: torch.Generator, lo: int, hi: int, n: int) -> np.ndarray:
    """floor(exp(U(ln lo, ln(hi+1)))) clamped to [lo, hi]."""
    u = torch.rand((n,), generator=gen, dtype=torch.float64).numpy()
    x = np.floor(np.exp(np.log(lo) + u * (np.log(hi + 1) - np.log(lo))))
    return np.clip(x, lo, hi).astype(np.int64)


def _blocks(n_tokens: int, bs: int) -> int:
    return (int(n_tokens) + bs - 1) // bs


def _pool_blocks(prefix_lens, group_of_req, context_lens, bs, factor=1.5):
    live = sum(_blocks(p, bs) for p in prefix_lens)
    for r in range(len(context_lens)):
        g = int(group_of_req[r])
        p = 0 if g < 0 else prefix_lens[g]
        live += _blocks(context_lens[r], bs) - p // bs
    return int(math.ceil(factor * live))


def _shapes(name: str, gen: torch.Generator, scale_requests: float = 1.0):
    """Lengths for each named workload.  Returns a dict of host arrays."""
    bs = BLOCK_SIZE
    if name == "tiny":
        # 8 q / 2 kv heads, d 64; 4 requests share a 256-token prefix; private
        # suffixes of 32/48/64/96 tokens are prefilled this step.
        suf = np.array([32, 48, 64, 96], np.int64)
        R = 4
        return dict(Hq=8, Hkv=2, d=64, prefix_lens=[256],
                    group=np.zeros(R, np.int64), cached=np.full(R, 256, np.int64),
                    new=suf, decode=np.zeros(R, bool), num_blocks=64)
    if name == "tiny_decode":
        # the tiny batch one step later: the suffix is cached and one token is
        # decoded per request (L = 289/305/321/353)
        suf = np.array([32, 48, 64, 96], np.int64)
        R = 4
        return dict(Hq=8, Hkv=2, d=64, prefix_lens=[256],
                    group=np.zeros(R, np.int64), cached=256 + suf,
                    new=np.ones(R, np.int64), decode=np.ones(R, bool), num_blocks=64)
    if name == "l8b_decode":
        R = max(1, int(round(64 * scale_requests)))
        suf = _uniform_int(gen, 256, 1024, R)
        gen_t = _uniform_int(gen, 0, 128, R)
        P = 4096
        return dict(Hq=32, Hkv=8, d=128, prefix_lens=[P], group=np.zeros(R, np.int64),
                    cached=P + suf + gen_t, new=np.ones(R, np.int64),
                    decode=np.ones(R, bool), num_blocks=None)
    if name == "l8b_prefill":
        R = max(1, int(round(32 * scale_requests)))
        S = _uniform_int(gen, 512, 1024, R)
        P = 4096
        return dict(Hq=32, Hkv=8, d=128, prefix_lens=[P], group=np.zeros(R, np.int64),
                    cached=np.full(R, P, np.int64), new=S,
                    decode=np.zeros(R, bool), num_blocks=None)
    if name == "qwen_mixed":
        Rd = max(3, int(round(256 * scale_requests)))
        Rp = max(1, int(round(8 * scale_requests)))
        prefixes = [2048, 4096, 6144]
        grp_d = (3 * np.arange(Rd)) // Rd            # contiguous thirds
        suf = _uniform_int(gen, 128, 1024, Rd)
        gen_t = _uniform_int(gen, 0, 64, Rd)
        cached_d = np.array([prefixes[g] for g in grp_d], np.int64) + suf + gen_t
        j = np.arange(Rp)
        grp_p = j % 3
        cached_p = np.array([prefixes[g] for g in grp_p], np.int64) + 512 * (j % 3)
        return dict(Hq=28, Hkv=4, d=128, prefix_lens=prefixes,
                    group=np.concatenate([grp_d, grp_p]),
                    cached=np.concatenate([cached_d, cached_p]),
                    new=np.concatenate([np.ones(Rd, np.int64), np.full(Rp, 512, np.int64)]),
                    decode=np.concatenate([np.ones(Rd, bool), np.zeros(Rp, bool)]),
                    num_blocks=None)
    if name == "l70b_decode":
        R = max(1, int(round(512 * scale_requests)))
        suf = _log_uniform_int(gen, 64, 2048, R)
        gen_t = _uniform_int(gen, 0, 128, R)
        P = 6144
        return dict(Hq=64, Hkv=8, d=128, prefix_lens=[P], group=np.zeros(R, np.int64),
                    cached=P + suf + gen_t, new=np.ones(R, np.int64),
                    decode=np.ones(R, bool), num_blocks=None)
    raise ValueError(f"unknown workload {name!r}")


def make_workload(name: str, seed: int | None = None, scale_requests: float = 1.0,
                  values: bool = True, custom: dict | None = None) -> Workload:
    """Build a named workload (or ``custom`` shapes) with seeded values.

    ``scale_requests`` shrinks the request count (parity tests at sizes the
    oracle finishes quickly); ``values=False`` skips the random tensors.
    ``custom`` is a dict with keys Hq, Hkv, d, prefix_lens, group, cached, new,
    decode and optionally num_blocks.
    """
    if seed is None:
        base = name.replace("_decode", "") if name == "tiny_decode" else name
        idx = WORKLOAD_NAMES.index(base) if base in WORKLOAD_NAMES else 99
        seed = BASE_SEED + idx
    gen = torch.Generator().manual_seed(int(seed))
    sh = dict(custom) if custom is not None else _shapes(name, gen, scale_requests)
    bs = BLOCK_SIZE
    group = np.asarray(sh["group"], np.int32)
    cached = np.asarray(sh["cached"], np.int32)
    new = np.asarray(sh["new"], np.int32)
    decode = np.asarray(sh["decode"], bool)
    prefix_lens = [int(p) for p in sh["prefix_lens"]]
    for p in prefix_lens:
        assert p % bs == 0, "shared prefixes are whole blocks"
    ctx = cached + new
    num_blocks = sh.get("num_blocks")
    if num_blocks is None:
        num_blocks = _pool_blocks(prefix_lens, group, ctx, bs)
    placement_seed = int(torch.randint(1, 2**62, (1,), generator=gen).item())
    Hq, Hkv, d = int(sh["Hq"]), int(sh["Hkv"]), int(sh["d"])
    R = len(cached)
    cu_new = np.zeros(R + 1, np.int64)
    cu_new[1:] = np.cumsum(new)
    priv_len = np.array([cached[r] - (prefix_lens[group[r]] if group[r] >= 0 else 0)
                         for r in range(R)], np.int64)
    priv_off = np.zeros(R + 1, np.int64)
    priv_off[1:] = np.cumsum(priv_len)
    w = Workload(name=name, seed=int(seed), num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d,
                 block_size=bs, prefix_lens=prefix_lens, group_of_req=group,
                 cached_lens=cached, new_lens=new, is_decode=decode,
                 num_blocks=int(num_blocks), placement_seed=placement_seed,
                 priv_off=priv_off, cu_new=cu_new)
    if not values:
        return w
    for p in prefix_lens:
        w.prefix_k.append(_randn_bf16(gen, (p, Hkv, d)))
        w.prefix_v.append(_randn_bf16(gen, (p, Hkv, d)))
    total_priv = int(priv_off[-1])
    w.priv_k = torch.empty((total_priv, Hkv, d), dtype=torch.bfloat16)
    w.priv_v = torch.empty((total_priv, Hkv, d), dtype=torch.bfloat16)
    for r in range(R):
        a, b = int(priv_off[r]), int(priv_off[r + 1])
        w.priv_k[a:b] = _randn_bf16(gen, (b - a, Hkv, d))
        w.priv_v[a:b] = _randn_bf16(gen, (b - a, Hkv, d))
    T = int(cu_new[-1])
    w.new_k = _randn_bf16(gen, (T, Hkv, d))
    w.new_v = _randn_bf16(gen, (T, Hkv, d))
    w.q = _randn_bf16(gen, (T, Hq, d))
    return w


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """The raw bf16 bit patterns of a CPU tensor as a uint16 numpy array."""
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)
