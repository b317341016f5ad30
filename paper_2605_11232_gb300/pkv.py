"""ctypes binding of ``libpkv.so`` (include/pkv.h), argument marshalling only.

Every function here forwards to the C entry point of the same name.  Device
buffers are torch CUDA tensors owned by the caller; host arrays are numpy.
There is no fallback: if the library cannot be loaded, every call raises.

The C entry points take bare device pointers, so they cannot see a tensor of
the wrong dtype or with too few rows.  The wrappers of the kernel calls
therefore check each tensor's dtype and shape against the layout the entry
point reads (ValueError) before any pointer is taken: a mismatch that would
make a kernel read or write past a buffer is refused on the host.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libpkv.so")

PKV_OK = 0
PKV_ERR_INVALID_ARG = -1
PKV_ERR_OUT_OF_BLOCKS = -2
PKV_ERR_REFCOUNT = -3
PKV_ERR_SHARED_BLOCK_WRITE = -4
PKV_ERR_CUDA = -5
PKV_ERR_UNSUPPORTED = -6
PKV_ERR_WORKSPACE = -7
PKV_ERR_DEVICE_TIMEOUT = -8
PKV_ERR_DEVICE_BOUNDS = -9
PKV_DTYPE_BF16 = 1

# every entry point declared in include/pkv.h
EXPORTS = [
    "kv_pool_create", "kv_pool_destroy", "kv_pool_alloc", "kv_pool_retain", "kv_pool_release",
    "kv_pool_refcount", "kv_pool_num_free", "kv_pool_alloc_sequence", "kv_slot_mapping",
    "kv_cache_write", "paged_attn_prefill", "paged_attn_decode_workspace_size",
    "paged_attn_decode", "paged_attn_decode_append", "paged_attn_decode_noalloc", "paged_attn_decode_step", "pkv_trace_enable",
    "pkv_trace_read", "pkv_check_device_errors", "pkv_last_error", "pkv_prefix_cache_create",
    "pkv_prefix_cache_destroy", "pkv_prefix_cache_match", "pkv_prefix_cache_insert",
    "pkv_prefix_cache_evict", "pkv_prefix_cache_size", "pkv_prefix_groups_build",
    "pkv_selftest_wait_timeout", "pkv_lora_dispatch", "pkv_check_block_table",
    "paged_attn_verify_tree", "pkv_tree_masks", "pkv_blocks_staging_size", "pkv_blocks_gather",
    "pkv_blocks_scatter", "pkv_lora_sgmv", "paged_attn_prefill_append",
    "paged_attn_verify_tree_workspace_size", "paged_attn_verify_tree_grouped", "pkv_verify_groups_build",
]


class PkvError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"pkv error {code}: {msg}")
        self.code = code


class PoolDesc(ctypes.Structure):
    _fields_ = [("num_blocks", ctypes.c_int32), ("block_size", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("placement_seed", ctypes.c_uint64)]


class KernelTime(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("total_ms", ctypes.c_double)]


class PrefixGroups(ctypes.Structure):
    _fields_ = [("num_groups", ctypes.c_int32), ("max_group_blocks", ctypes.c_int32),
                ("max_group_members", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("group_start", ctypes.c_void_p), ("member_req", ctypes.c_void_p),
                ("group_blocks", ctypes.c_void_p), ("group_of_req", ctypes.c_void_p)]


class VerifyGroups(ctypes.Structure):
    _fields_ = [("num_groups", ctypes.c_int32), ("max_group_blocks", ctypes.c_int32),
                ("max_group_tokens", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("group_start", ctypes.c_void_p), ("member_token", ctypes.c_void_p),
                ("group_blocks", ctypes.c_void_p), ("group_row", ctypes.c_void_p),
                ("request_group", ctypes.c_void_p)]


class StepLayout(ctypes.Structure):
    """Byte offsets of one decode step's inputs in a packed buffer (pkv_step_layout)."""
    _fields_ = [("q", ctypes.c_size_t), ("k_new", ctypes.c_size_t), ("v_new", ctypes.c_size_t),
                ("slot_mapping", ctypes.c_size_t), ("context_lens", ctypes.c_size_t),
                ("bytes", ctypes.c_size_t), ("flags", ctypes.c_uint64)]


PKV_STEP_FUSED_WRITE = 1


_lib = None


def load(path: str | None = None):
    """Load the library (built by ``__graft_entry__.build()`` / ``build.py``)."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libpkv.so not built ({p}); run __graft_entry__.build()")
    lib = ctypes.CDLL(p)
    V, P, i32, i64, f32 = (ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                           ctypes.c_float)
    sz = ctypes.c_size_t
    sig = {
        "kv_pool_create": [ctypes.POINTER(PoolDesc), V, V, ctypes.POINTER(V)],
        "kv_pool_destroy": [V],
        "kv_pool_alloc": [V, i32, P],
        "kv_pool_retain": [V, P, i32],
        "kv_pool_release": [V, P, i32],
        "kv_pool_refcount": [V, i32, P],
        "kv_pool_num_free": [V, P],
        "kv_pool_alloc_sequence": [V, P, i32, i32, P],
        "kv_slot_mapping": [V, P, i32, P, P, i32, P],
        "kv_cache_write": [V, V, V, V, i32, V],
        "paged_attn_prefill": [V, V, V, V, V, V, V, i32, i32, i32, i32, f32, V],
        "paged_attn_decode_workspace_size": [V, i32, i32, i32, ctypes.POINTER(PrefixGroups),
                                             ctypes.POINTER(sz)],
        "paged_attn_decode": [V, V, V, V, V, V, i32, i32, i32, f32,
                              ctypes.POINTER(PrefixGroups), V, sz, V],
        "paged_attn_decode_append": [V, V, V, V, V, V, V, V, i32, i32, i32, f32,
                                     ctypes.POINTER(PrefixGroups), V, sz, V],
        "pkv_check_device_errors": [V, V, P],
        "paged_attn_decode_noalloc": [V, V, V, V, V, V, i32, i32, i32, f32,
                                      ctypes.POINTER(PrefixGroups), V],
        "paged_attn_decode_step": [V, V, V, ctypes.POINTER(StepLayout), i32, V, i32, i32, i32, f32,
                                   ctypes.POINTER(PrefixGroups), V, sz, V, V, V, V, V, V, V],
        "pkv_trace_enable": [V, i32],
        "pkv_prefix_cache_create": [V, i32, ctypes.POINTER(V)],
        "pkv_prefix_cache_destroy": [V],
        "pkv_prefix_cache_match": [V, P, i32, P, i32, P],
        "pkv_prefix_cache_insert": [V, P, i32, P, i32, P],
        "pkv_prefix_cache_evict": [V, i32, P, P],
        "pkv_prefix_cache_size": [V, P],
        "pkv_prefix_groups_build": [P, i32, i32, P, i32, P, P, P, P, P, P, P],
        "pkv_selftest_wait_timeout": [V, i32, V],
        "pkv_lora_dispatch": [P, P, i32, P, i32, i32, P, P, P, P, P],
        "pkv_check_block_table": [V, P, i32, i32, P, P],
        "paged_attn_verify_tree": [V, V, V, V, V, V, V, i32, i32, i32, i32, f32, V, V],
        "pkv_tree_masks": [P, P, i32, P],
        "paged_attn_verify_tree_workspace_size": [V, i32, i32, i32, ctypes.POINTER(VerifyGroups),
                                                  ctypes.POINTER(sz)],
        "paged_attn_verify_tree_grouped": [V, V, V, V, V, V, V, i32, i32, i32, i32, i32, f32, V,
                                           ctypes.POINTER(VerifyGroups), V, sz, V],
        "pkv_verify_groups_build": [P, P, i32, i32, P, P, P, P],
        "pkv_blocks_staging_size": [V, i32, ctypes.POINTER(sz)],
        "paged_attn_prefill_append": [V, V, V, V, i32, V, V, V, V, V, i32, i32, i32, i32, f32, V],
        "pkv_lora_sgmv": [V, V, V, V, P, P, P, i32, i32, i32, i32, i32, i32, V, V, V],
        "pkv_blocks_gather": [V, V, i32, V, V],
        "pkv_blocks_scatter": [V, V, i32, V, V],
        "pkv_trace_read": [V, P, i32, P],
    }
    for name, args in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    lib.pkv_last_error.argtypes = []
    lib.pkv_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(rc: int):
    if rc != PKV_OK:
        raise PkvError(rc, load().pkv_last_error().decode())


def _np_ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dptr(t):
    """Device address of a torch tensor (or None)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


# (num_blocks, num_kv_heads, head_dim) of every pool this module created
_POOL_GEOMETRY: dict = {}


def _need(cond, msg):
    """Raise ValueError unless cond; msg is a string or a callable that makes
    one (so that a passing check formats nothing)."""
    if not cond:
        raise ValueError(msg() if callable(msg) else msg)


def _pool_geometry(pool):
    key = pool.value if isinstance(pool, ctypes.c_void_p) else pool
    return _POOL_GEOMETRY.get(key)


def _check_tensor(name, t, dtype, ndim):
    """The tensor's shape, after checking that it exists, has this dtype and
    this many dimensions."""
    if t is None:
        raise ValueError(f"{name} is required")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    shape = t.shape
    if len(shape) != ndim:
        raise ValueError(f"{name} must have {ndim} dimensions, got shape {tuple(shape)}")
    return shape


def _check_cache_write_args(pool, k_new, v_new, slot_mapping):
    """k_new, v_new bf16 [>= T][Hkv][d]; slot_mapping int64 [T]."""
    import torch
    T = _check_tensor("slot_mapping", slot_mapping, torch.int64, 1)[0]
    geo = _pool_geometry(pool)
    for name, t in (("k_new", k_new), ("v_new", v_new)):
        ts = _check_tensor(name, t, torch.bfloat16, 3)
        _need(ts[0] >= T, lambda: f"{name} has {ts[0]} rows for {T} slots")
        if geo is not None:
            _need(ts[1] == geo[1] and ts[2] == geo[2],
                  lambda: f"{name} rows must be [num_kv_heads][head_dim] = {list(geo[1:])}, "
                  f"got {list(ts[1:])}")


def _check_attn_args(pool, q, out, lse, context_lens, block_table, min_q_rows):
    """q bf16 [>= min_q_rows][Hq][d] with d the pool's head dim and Hq a
    multiple of its kv heads; out bf16 with q's row layout; lse fp32 [.][Hq]
    or None; context_lens int32 [R]; block_table int32 [>= R][max_blocks]."""
    import torch
    R = _check_tensor("context_lens", context_lens, torch.int32, 1)[0]
    bs = _check_tensor("block_table", block_table, torch.int32, 2)
    _need(bs[0] >= R, lambda: f"block_table has {bs[0]} rows for {R} requests")
    _need(bs[1] >= 1, "block_table needs at least one column")
    qs = _check_tensor("q", q, torch.bfloat16, 3)
    _need(qs[0] >= min_q_rows, lambda: f"q has {qs[0]} rows, {min_q_rows} needed")
    geo = _pool_geometry(pool)
    if geo is not None:
        _need(qs[2] == geo[2], lambda: f"q head dim {qs[2]} != the pool's {geo[2]}")
        _need(qs[1] % geo[1] == 0,
              lambda: f"{qs[1]} query heads are not a multiple of the pool's {geo[1]} kv heads")
    os_ = _check_tensor("out", out, torch.bfloat16, 3)
    _need(os_[1] == qs[1] and os_[2] == qs[2],
          lambda: f"out rows must be {list(qs[1:])}, got {list(os_[1:])}")
    _need(os_[0] >= min_q_rows, lambda: f"out has {os_[0]} rows, {min_q_rows} needed")
    if lse is not None:
        ls = _check_tensor("lse", lse, torch.float32, 2)
        _need(ls[1] == qs[1], lambda: f"lse must have {qs[1]} columns, got {ls[1]}")
        _need(ls[0] >= min_q_rows, lambda: f"lse has {ls[0]} rows, {min_q_rows} needed")


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


# ---- a1: pool ---------------------------------------------------------------

def kv_pool_create(num_blocks: int, num_kv_heads: int, head_dim: int, k_cache=None,
                   v_cache=None, placement_seed: int = 0, block_size: int = 16):
    desc = PoolDesc(num_blocks, block_size, num_kv_heads, head_dim, PKV_DTYPE_BF16, 0,
                    placement_seed & (2**64 - 1))
    if k_cache is not None or v_cache is not None:
        import torch
        shape = (num_blocks, num_kv_heads, block_size, head_dim)
        for name, t in (("k_cache", k_cache), ("v_cache", v_cache)):
            _check_tensor(name, t, torch.bfloat16, 4)
            _need(tuple(t.shape) == shape, lambda: f"{name} must have shape {list(shape)}, got {list(t.shape)}")
    h = ctypes.c_void_p()
    _check(load().kv_pool_create(ctypes.byref(desc), _dptr(k_cache), _dptr(v_cache),
                                 ctypes.byref(h)))
    _POOL_GEOMETRY[h.value] = (int(num_blocks), int(num_kv_heads), int(head_dim))
    return h


def kv_pool_destroy(pool):
    _check(load().kv_pool_destroy(pool))
    _POOL_GEOMETRY.pop(pool.value if isinstance(pool, ctypes.c_void_p) else pool, None)


def kv_pool_alloc(pool, n: int) -> np.ndarray:
    ids = np.zeros(max(n, 1), np.int32)
    _check(load().kv_pool_alloc(pool, n, _np_ptr(ids)))
    return ids[:n]


def kv_pool_retain(pool, ids):
    ids = np.ascontiguousarray(ids, np.int32)
    _check(load().kv_pool_retain(pool, _np_ptr(ids), len(ids)))


def kv_pool_release(pool, ids):
    ids = np.ascontiguousarray(ids, np.int32)
    _check(load().kv_pool_release(pool, _np_ptr(ids), len(ids)))


def kv_pool_refcount(pool, block_id: int) -> int:
    out = np.zeros(1, np.int32)
    _check(load().kv_pool_refcount(pool, int(block_id), _np_ptr(out)))
    return int(out[0])


def kv_pool_num_free(pool) -> int:
    out = np.zeros(1, np.int32)
    _check(load().kv_pool_num_free(pool, _np_ptr(out)))
    return int(out[0])


def kv_pool_alloc_sequence(pool, prefix_ids, n_blocks: int) -> np.ndarray:
    pre = np.ascontiguousarray(prefix_ids if prefix_ids is not None else [], np.int32)
    row = np.zeros(max(n_blocks, 1), np.int32)
    _check(load().kv_pool_alloc_sequence(pool, _np_ptr(pre) if len(pre) else None, len(pre),
                                         int(n_blocks), _np_ptr(row)))
    return row[:n_blocks]


# ---- a2: slot mapping --------------------------------------------------------

def kv_slot_mapping(pool, block_table: np.ndarray, context_lens, new_lens,
                    out: np.ndarray | None = None) -> np.ndarray:
    """Slots of the new tokens; written into ``out`` (contiguous int64, one per
    new token) when given, e.g. a view of a pinned step buffer."""
    table = np.ascontiguousarray(block_table, np.int32)
    ctx = np.ascontiguousarray(context_lens, np.int32)
    new = np.ascontiguousarray(new_lens, np.int32)
    n = int(new.sum())
    if out is None:
        out = np.zeros(max(n, 1), np.int64)
    elif out.dtype != np.int64 or not out.flags.c_contiguous or out.size < n:
        raise ValueError("out must be a contiguous int64 array with one entry per new token")
    _check(load().kv_slot_mapping(pool, _np_ptr(table), table.shape[1], _np_ptr(ctx),
                                  _np_ptr(new), len(ctx), _np_ptr(out)))
    return out[:n]


def pkv_check_block_table(pool, block_table, context_lens) -> None:
    """Raise PkvError (with .bad_request) unless every table entry a kernel
    will read names an allocated block of the pool."""
    table = np.ascontiguousarray(block_table, np.int32)
    ctx = np.ascontiguousarray(context_lens, np.int32)
    if table.ndim != 2 or table.shape[0] != len(ctx):
        raise ValueError("block_table must be [num_requests][max_blocks]")
    bad = np.zeros(1, np.int32)
    rc = load().pkv_check_block_table(pool, _np_ptr(table), table.shape[1], len(ctx), _np_ptr(ctx),
                                      _np_ptr(bad))
    if rc != PKV_OK:
        err = PkvError(rc, pkv_last_error())
        err.bad_request = int(bad[0])
        raise err


# ---- a3-a7: kernels ---------------------------------------------------------

def kv_cache_write(pool, k_new, v_new, slot_mapping, stream=None):
    _check_cache_write_args(pool, k_new, v_new, slot_mapping)
    _check(load().kv_cache_write(pool, _dptr(k_new), _dptr(v_new), _dptr(slot_mapping),
                                 int(slot_mapping.shape[0]), _stream(stream)))


def paged_attn_prefill(pool, q, out, lse, cu_seqlens_q, context_lens, block_table,
                       max_seqlen_q: int, scale: float, stream=None):
    import torch
    _check_attn_args(pool, q, out, lse, context_lens, block_table, 0)
    _need(tuple(out.shape) == tuple(q.shape), lambda: f"out must have q's shape {list(q.shape)}")
    if lse is not None:
        _need(lse.shape[0] == q.shape[0], lambda: f"lse must have {q.shape[0]} rows")
    _check_tensor("cu_seqlens_q", cu_seqlens_q, torch.int32, 1)
    _need(cu_seqlens_q.shape[0] == context_lens.shape[0] + 1,
          lambda: f"cu_seqlens_q must have {context_lens.shape[0] + 1} entries")
    _check(load().paged_attn_prefill(
        pool, _dptr(q), _dptr(out), _dptr(lse), _dptr(cu_seqlens_q), _dptr(context_lens),
        _dptr(block_table), int(block_table.shape[1]), int(context_lens.shape[0]),
        int(max_seqlen_q), int(q.shape[1]), float(scale), _stream(stream)))


def paged_attn_prefill_append(pool, q, k_new, v_new, out, lse, cu_seqlens_q, context_lens, block_table,
                              max_seqlen_q: int, scale: float, stream=None):
    """paged_attn_prefill with the new tokens' K/V (bf16 [T][Hkv][d], rows in
    q's order) stored into the pool by the prefill kernel."""
    import torch
    _check_attn_args(pool, q, out, lse, context_lens, block_table, 0)
    _need(tuple(out.shape) == tuple(q.shape), lambda: f"out must have q's shape {list(q.shape)}")
    if lse is not None:
        _need(lse.shape[0] == q.shape[0], lambda: f"lse must have {q.shape[0]} rows")
    _check_tensor("cu_seqlens_q", cu_seqlens_q, torch.int32, 1)
    _need(cu_seqlens_q.shape[0] == context_lens.shape[0] + 1,
          lambda: f"cu_seqlens_q must have {context_lens.shape[0] + 1} entries")
    T = int(q.shape[0])
    geo = _pool_geometry(pool)
    for name, t in (("k_new", k_new), ("v_new", v_new)):
        ts = _check_tensor(name, t, torch.bfloat16, 3)
        _need(ts[0] == T, lambda: f"{name} must have q's {T} rows, got {ts[0]}")
        if geo is not None:
            _need(ts[1] == geo[1] and ts[2] == geo[2],
                  lambda: f"{name} rows must be [{geo[1]}][{geo[2]}], got {list(ts[1:])}")
    _check(load().paged_attn_prefill_append(
        pool, _dptr(q), _dptr(k_new), _dptr(v_new), T, _dptr(out), _dptr(lse), _dptr(cu_seqlens_q),
        _dptr(context_lens), _dptr(block_table), int(block_table.shape[1]), int(context_lens.shape[0]),
        int(max_seqlen_q), int(q.shape[1]), float(scale), _stream(stream)))


def paged_attn_verify_tree(pool, q, out, lse, cu_seqlens_q, context_lens, block_table,
                           max_seqlen_q: int, scale: float, tree_mask, stream=None):
    """paged_attn_prefill over tree-shaped drafts: tree_mask is a device
    int64 tensor [T] of draft masks (pkv_tree_masks)."""
    import torch
    _check_attn_args(pool, q, out, lse, context_lens, block_table, 0)
    _need(tuple(out.shape) == tuple(q.shape), lambda: f"out must have q's shape {list(q.shape)}")
    cs = _check_tensor("cu_seqlens_q", cu_seqlens_q, torch.int32, 1)
    _need(cs[0] == context_lens.shape[0] + 1,
          lambda: f"cu_seqlens_q must have {context_lens.shape[0] + 1} entries")
    ms = _check_tensor("tree_mask", tree_mask, torch.int64, 1)
    _need(ms[0] >= q.shape[0], lambda: f"tree_mask has {ms[0]} entries for {q.shape[0]} rows")
    _check(load().paged_attn_verify_tree(
        pool, _dptr(q), _dptr(out), _dptr(lse), _dptr(cu_seqlens_q), _dptr(context_lens),
        _dptr(block_table), int(block_table.shape[1]), int(context_lens.shape[0]),
        int(max_seqlen_q), int(q.shape[1]), float(scale), _dptr(tree_mask), _stream(stream)))


def pkv_verify_groups_build(cu_seqlens, request_group, num_groups: int) -> dict:
    """Token groups of a verification batch (host): a dict with group_start,
    member_token, group_row (int32 numpy arrays) and max_group_tokens."""
    cu = np.ascontiguousarray(cu_seqlens, np.int32)
    rg = np.ascontiguousarray(request_group, np.int32)
    R = len(cu) - 1
    _need(len(rg) == R, lambda: f"request_group must have {R} entries")
    G = int(num_groups)
    gstart = np.zeros(G + 1, np.int32)
    members = np.zeros(max(int(cu[-1]), 1), np.int32)
    grow = np.zeros(max(G, 1), np.int32)
    mx = np.zeros(1, np.int32)
    _check(load().pkv_verify_groups_build(_np_ptr(cu), _np_ptr(rg), R, G, _np_ptr(gstart), _np_ptr(members),
                                          _np_ptr(grow), _np_ptr(mx)))
    return dict(group_start=gstart, member_token=members[:int(gstart[G])], group_row=grow[:G],
                max_group_tokens=int(mx[0]))


def make_verify_groups(num_groups=0, max_group_blocks=0, max_group_tokens=0, group_start=None,
                       member_token=None, group_blocks=None, group_row=None, request_group=None):
    """The pkv_verify_groups descriptor over device int32 tensors (they must
    outlive every call that takes it)."""
    import torch
    for name, t, n in (("group_start", group_start, num_groups + 1), ("member_token", member_token, 0),
                       ("group_blocks", group_blocks, num_groups), ("group_row", group_row, num_groups),
                       ("request_group", request_group, 0)):
        if t is not None or num_groups > 0:
            _check_tensor(name, t, torch.int32, 1)
            _need(t.shape[0] >= n, lambda: f"{name} has {t.shape[0]} entries, {n} needed")
    return VerifyGroups(int(num_groups), int(max_group_blocks), int(max_group_tokens), 0,
                        _dptr(group_start), _dptr(member_token), _dptr(group_blocks), _dptr(group_row),
                        _dptr(request_group))


def paged_attn_verify_tree_workspace_size(pool, num_tokens: int, num_q_heads: int, max_blocks: int,
                                          groups=None) -> int:
    out = ctypes.c_size_t()
    _check(load().paged_attn_verify_tree_workspace_size(
        pool, int(num_tokens), int(num_q_heads), int(max_blocks),
        ctypes.byref(groups) if groups is not None else None, ctypes.byref(out)))
    return int(out.value)


def paged_attn_verify_tree_grouped(pool, q, out, lse, cu_seqlens_q, context_lens, block_table,
                                   max_seqlen_q: int, scale: float, tree_mask, groups, workspace,
                                   stream=None):
    """paged_attn_verify_tree with each group's shared prefix read once per
    group (groups: make_verify_groups(...) or None)."""
    import torch
    _check_attn_args(pool, q, out, lse, context_lens, block_table, 0)
    _need(tuple(out.shape) == tuple(q.shape), lambda: f"out must have q's shape {list(q.shape)}")
    cs = _check_tensor("cu_seqlens_q", cu_seqlens_q, torch.int32, 1)
    _need(cs[0] == context_lens.shape[0] + 1,
          lambda: f"cu_seqlens_q must have {context_lens.shape[0] + 1} entries")
    ms = _check_tensor("tree_mask", tree_mask, torch.int64, 1)
    _need(ms[0] >= q.shape[0], lambda: f"tree_mask has {ms[0]} entries for {q.shape[0]} rows")
    _check(load().paged_attn_verify_tree_grouped(
        pool, _dptr(q), _dptr(out), _dptr(lse), _dptr(cu_seqlens_q), _dptr(context_lens),
        _dptr(block_table), int(block_table.shape[1]), int(context_lens.shape[0]), int(q.shape[0]),
        int(max_seqlen_q), int(q.shape[1]), float(scale), _dptr(tree_mask),
        ctypes.byref(groups) if groups is not None else None, _dptr(workspace),
        int(workspace.numel() * workspace.element_size()) if workspace is not None else 0,
        _stream(stream)))


def pkv_blocks_staging_size(pool, n: int) -> int:
    out = ctypes.c_size_t(0)
    _check(load().pkv_blocks_staging_size(pool, int(n), ctypes.byref(out)))
    return int(out.value)


def _check_transfer_args(pool, block_ids, staging):
    import torch
    n = _check_tensor("block_ids", block_ids, torch.int32, 1)[0]
    nbytes = staging.numel() * staging.element_size()
    need = pkv_blocks_staging_size(pool, n)
    _need(staging.is_cuda and staging.is_contiguous() and nbytes >= need,
          lambda: f"staging must be a contiguous device buffer of >= {need} bytes, got {nbytes}")
    return n


def pkv_blocks_gather(pool, block_ids, staging, stream=None):
    """Copy the pool's blocks block_ids (device int32 [n]) into staging."""
    n = _check_transfer_args(pool, block_ids, staging)
    _check(load().pkv_blocks_gather(pool, _dptr(block_ids), n, _dptr(staging), _stream(stream)))


def pkv_blocks_scatter(pool, block_ids, staging, stream=None):
    """Copy staging into the pool's blocks block_ids (device int32 [n])."""
    n = _check_transfer_args(pool, block_ids, staging)
    _check(load().pkv_blocks_scatter(pool, _dptr(block_ids), n, _dptr(staging), _stream(stream)))


def pkv_lora_sgmv(x, w, lora_a, lora_b, scale, seg_start, seg_adapter, y, error_word=None,
                  stream=None):
    """y = W x + s_a B_a (A_a x) per segment (device bf16 tensors; scale,
    seg_start, seg_adapter host arrays)."""
    import torch
    T, d_in = _check_tensor("x", x, torch.bfloat16, 2)
    d_out, wi = _check_tensor("w", w, torch.bfloat16, 2)
    _need(wi == d_in, lambda: f"w must be [d_out][{d_in}], got {list(w.shape)}")
    n_ad, rank, ai = _check_tensor("lora_a", lora_a, torch.bfloat16, 3)
    _need(ai == d_in, lambda: f"lora_a must be [n][rank][{d_in}], got {list(lora_a.shape)}")
    bs = _check_tensor("lora_b", lora_b, torch.bfloat16, 3)
    _need(tuple(bs) == (n_ad, d_out, rank), lambda: f"lora_b must be [{n_ad}][{d_out}][{rank}], got {list(bs)}")
    ys = _check_tensor("y", y, torch.bfloat16, 2)
    _need(tuple(ys) == (T, d_out), lambda: f"y must be [{T}][{d_out}], got {list(ys)}")
    for name, t in (("x", x), ("w", w), ("lora_a", lora_a), ("lora_b", lora_b), ("y", y)):
        _need(t.is_cuda and t.is_contiguous(), lambda: f"{name} must be a contiguous device tensor")
    sc = np.ascontiguousarray(scale, np.float32)
    st = np.ascontiguousarray(seg_start, np.int32)
    sa = np.ascontiguousarray(seg_adapter, np.int32)
    _need(len(sc) >= n_ad, lambda: f"scale needs {n_ad} entries")
    _need(len(st) == len(sa) + 1, "seg_start must have one entry more than seg_adapter")
    _check(load().pkv_lora_sgmv(_dptr(x), _dptr(w), _dptr(lora_a), _dptr(lora_b), _np_ptr(sc), _np_ptr(st),
                                _np_ptr(sa), len(sa), int(T), int(d_in), int(d_out), int(rank), int(n_ad),
                                _dptr(y), _dptr(error_word), _stream(stream)))


def pkv_tree_masks(parent, cu_seqlens) -> np.ndarray:
    """Draft masks (int64 view of the uint64 bits) of tree-shaped drafts."""
    par = np.ascontiguousarray(parent, np.int32)
    cu = np.ascontiguousarray(cu_seqlens, np.int32)
    out = np.zeros(max(len(par), 1), np.uint64)
    _check(load().pkv_tree_masks(_np_ptr(par), _np_ptr(cu), len(cu) - 1, _np_ptr(out)))
    return out[:len(par)].view(np.int64)


def make_prefix_groups(num_groups=0, max_group_blocks=0, max_group_members=0, group_start=None,
                       member_req=None, group_blocks=None, group_of_req=None):
    import torch
    for name, t, n in (("group_start", group_start, num_groups + 1), ("member_req", member_req, 0),
                       ("group_blocks", group_blocks, num_groups), ("group_of_req", group_of_req, 0)):
        if t is not None or num_groups > 0:
            _check_tensor(name, t, torch.int32, 1)
            _need(t.shape[0] >= n, lambda: f"{name} has {t.shape[0]} entries, {n} needed")
    return PrefixGroups(int(num_groups), int(max_group_blocks), int(max_group_members), 0,
                        _dptr(group_start), _dptr(member_req), _dptr(group_blocks),
                        _dptr(group_of_req))


def paged_attn_decode_workspace_size(pool, num_requests: int, num_q_heads: int,
                                     max_blocks: int, groups=None) -> int:
    out = ctypes.c_size_t()
    _check(load().paged_attn_decode_workspace_size(
        pool, int(num_requests), int(num_q_heads), int(max_blocks),
        ctypes.byref(groups) if groups is not None else None, ctypes.byref(out)))
    return int(out.value)


def paged_attn_decode(pool, q, out, lse, context_lens, block_table, scale: float, groups,
                      workspace, stream=None):
    _check_attn_args(pool, q, out, lse, context_lens, block_table, int(context_lens.shape[0]))
    _check(load().paged_attn_decode(
        pool, _dptr(q), _dptr(out), _dptr(lse), _dptr(context_lens), _dptr(block_table),
        int(block_table.shape[1]), int(context_lens.shape[0]), int(q.shape[1]), float(scale),
        ctypes.byref(groups) if groups is not None else None, _dptr(workspace),
        int(workspace.numel() * workspace.element_size()) if workspace is not None else 0,
        _stream(stream)))


def paged_attn_decode_append(pool, q, k_new, v_new, out, lse, context_lens, block_table, scale: float,
                             groups, workspace, stream=None):
    """paged_attn_decode with the query tokens' own K/V (bf16 [R][Hkv][d])
    stored into the pool by the decode kernels."""
    import torch
    R = int(context_lens.shape[0])
    _check_attn_args(pool, q, out, lse, context_lens, block_table, R)
    geo = _pool_geometry(pool)
    for name, t in (("k_new", k_new), ("v_new", v_new)):
        ts = _check_tensor(name, t, torch.bfloat16, 3)
        _need(ts[0] >= R, lambda: f"{name} has {ts[0]} rows, {R} needed")
        if geo is not None:
            _need(ts[1] == geo[1] and ts[2] == geo[2],
                  lambda: f"{name} rows must be [{geo[1]}][{geo[2]}], got {list(ts[1:])}")
    _check(load().paged_attn_decode_append(
        pool, _dptr(q), _dptr(k_new), _dptr(v_new), _dptr(out), _dptr(lse), _dptr(context_lens),
        _dptr(block_table), int(block_table.shape[1]), R, int(q.shape[1]), float(scale),
        ctypes.byref(groups) if groups is not None else None, _dptr(workspace),
        int(workspace.numel() * workspace.element_size()) if workspace is not None else 0,
        _stream(stream)))


def paged_attn_decode_noalloc(pool, q, out, lse, context_lens, block_table, scale: float,
                              groups, stream=None):
    """paged_attn_decode with the library's static scratch (no workspace)."""
    _check_attn_args(pool, q, out, lse, context_lens, block_table, int(context_lens.shape[0]))
    _check(load().paged_attn_decode_noalloc(
        pool, _dptr(q), _dptr(out), _dptr(lse), _dptr(context_lens), _dptr(block_table),
        int(block_table.shape[1]), int(context_lens.shape[0]), int(q.shape[1]), float(scale),
        ctypes.byref(groups) if groups is not None else None, _stream(stream)))


def _hptr(t):
    """Address of a host (CPU) torch tensor, or None."""
    if t is None:
        return None
    if t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CPU tensor")
    return ctypes.c_void_p(t.data_ptr())


def _event(ev):
    """cudaEvent_t of a torch.cuda.Event (created on first use), or None."""
    if ev is None:
        return None
    if ev.cuda_event == 0:
        ev.record()   # torch creates the CUDA event lazily, at its first record
    return ctypes.c_void_p(ev.cuda_event)


def _check_step_args(pool, host_in, dev_in, layout, block_table, num_q_heads, out, lse,
                     host_out, host_lse):
    """Both step buffers hold layout.bytes (the H2D copy moves that many);
    out bf16 [>= R][num_q_heads][d] and lse fp32 [>= R][num_q_heads] as the
    kernels write them; host_out / host_lse the same shape and dtype as the
    device tensors they receive."""
    import torch
    for name, t in (("host_in", host_in), ("dev_in", dev_in)):
        _need(t is not None, lambda: f"{name} is required")
        nbytes = t.numel() * t.element_size()
        _need(nbytes >= layout.bytes, lambda: f"{name} holds {nbytes} bytes, the layout needs {layout.bytes}")
    _check_tensor("block_table", block_table, torch.int32, 2)
    R = block_table.shape[0]
    _check_tensor("out", out, torch.bfloat16, 3)
    _need(out.shape[0] >= R and out.shape[1] == num_q_heads,
          lambda: f"out must be [>= {R}][{num_q_heads}][head_dim], got {list(out.shape)}")
    geo = _pool_geometry(pool)
    if geo is not None:
        _need(out.shape[2] == geo[2], lambda: f"out head dim {out.shape[2]} != the pool's {geo[2]}")
    if lse is not None:
        _check_tensor("lse", lse, torch.float32, 2)
        _need(lse.shape[0] >= R and lse.shape[1] == num_q_heads,
              lambda: f"lse must be [>= {R}][{num_q_heads}], got {list(lse.shape)}")
    for name, h, d in (("host_out", host_out, out), ("host_lse", host_lse, lse)):
        if h is not None:
            _need(d is not None, lambda: f"{name} needs its device tensor")
            _need(h.dtype == d.dtype and tuple(h.shape) == tuple(d.shape),
                  lambda: f"{name} must match its device tensor ({d.dtype} {list(d.shape)}), "
                  f"got {h.dtype} {list(h.shape)}")


def _step_args(pool, host_in, dev_in, layout, num_new_tokens, block_table, num_q_heads, scale,
               groups, workspace, out, lse, host_out, host_lse, wait_event, done_event, stream):
    _check_step_args(pool, host_in, dev_in, layout, block_table, num_q_heads, out, lse, host_out,
                     host_lse)
    return (pool, _hptr(host_in), _dptr(dev_in), ctypes.byref(layout), int(num_new_tokens),
            _dptr(block_table), int(block_table.shape[1]), int(block_table.shape[0]),
            int(num_q_heads), float(scale), ctypes.byref(groups) if groups is not None else None,
            _dptr(workspace),
            int(workspace.numel() * workspace.element_size()) if workspace is not None else 0,
            _dptr(out), _dptr(lse), _hptr(host_out), _hptr(host_lse), _event(wait_event),
            _event(done_event), _stream(stream))


def paged_attn_decode_step(pool, host_in, dev_in, layout: StepLayout, num_new_tokens: int,
                           block_table, num_q_heads: int, scale: float, groups, workspace, out,
                           lse=None, host_out=None, host_lse=None, wait_event=None,
                           done_event=None, stream=None):
    """One decode step from a packed host buffer (pinned uint8 CPU tensor):
    H2D copy, [wait for wait_event], cache write, decode, [record done_event],
    D2H copy of the output; enqueued, not waited for.  Events are
    torch.cuda.Event objects."""
    _check(load().paged_attn_decode_step(*_step_args(
        pool, host_in, dev_in, layout, num_new_tokens, block_table, num_q_heads, scale, groups,
        workspace, out, lse, host_out, host_lse, wait_event, done_event, stream)))


class DecodeStep:
    """paged_attn_decode_step with its arguments converted once, for a serving
    loop that calls it every step on the same buffers (keeps them alive)."""

    def __init__(self, pool, host_in, dev_in, layout: StepLayout, num_new_tokens: int,
                 block_table, num_q_heads: int, scale: float, groups, workspace, out, lse=None,
                 host_out=None, host_lse=None, wait_event=None, done_event=None, stream=None):
        self._keep = (host_in, dev_in, layout, block_table, groups, workspace, out, lse, host_out,
                      host_lse, wait_event, done_event, stream)
        self._args = _step_args(pool, host_in, dev_in, layout, num_new_tokens, block_table,
                                num_q_heads, scale, groups, workspace, out, lse, host_out,
                                host_lse, wait_event, done_event, stream)
        self._fn = load().paged_attn_decode_step

    def __call__(self):
        _check(self._fn(*self._args))


# ---- automatic prefix caching (host) ----------------------------------------

PKV_PREFIX_CACHE_WEAK_HASH = 1


def pkv_prefix_cache_create(pool, weak_hash: bool = False):
    h = ctypes.c_void_p()
    _check(load().pkv_prefix_cache_create(pool, PKV_PREFIX_CACHE_WEAK_HASH if weak_hash else 0,
                                          ctypes.byref(h)))
    return h


def pkv_prefix_cache_destroy(cache):
    _check(load().pkv_prefix_cache_destroy(cache))


def pkv_prefix_cache_match(cache, tokens, max_ids: int | None = None) -> np.ndarray:
    """Ids of the longest run of cached full blocks heading `tokens` (each
    retained once more for the caller)."""
    t = np.ascontiguousarray(tokens, np.int32)
    cap = len(t) // 16 if max_ids is None else int(max_ids)
    out = np.zeros(max(cap, 1), np.int32)
    n = np.zeros(1, np.int32)
    _check(load().pkv_prefix_cache_match(cache, _np_ptr(t), len(t), _np_ptr(out), cap, _np_ptr(n)))
    return out[: int(n[0])]


def pkv_prefix_cache_insert(cache, tokens, ids) -> int:
    """Register the full blocks of `tokens` held in `ids`; returns the number
    of new entries."""
    t = np.ascontiguousarray(tokens, np.int32)
    i = np.ascontiguousarray(ids, np.int32)
    n = np.zeros(1, np.int32)
    _check(load().pkv_prefix_cache_insert(cache, _np_ptr(t), len(t), _np_ptr(i), len(i), _np_ptr(n)))
    return int(n[0])


def pkv_prefix_cache_evict(cache, n_wanted: int) -> np.ndarray:
    out = np.zeros(max(int(n_wanted), 1), np.int32)
    n = np.zeros(1, np.int32)
    _check(load().pkv_prefix_cache_evict(cache, int(n_wanted), _np_ptr(out), _np_ptr(n)))
    return out[: int(n[0])]


def pkv_prefix_cache_size(cache) -> int:
    n = np.zeros(1, np.int32)
    _check(load().pkv_prefix_cache_size(cache, _np_ptr(n)))
    return int(n[0])


def pkv_prefix_groups_build(block_table, context_lens, min_shared_blocks: int = 1) -> dict:
    """Prefix groups of a decode batch from its host block tables: a dict with
    group_of_req, group_start, member_req, group_blocks (int32 numpy arrays),
    num_groups, max_group_blocks, max_group_members."""
    table = np.ascontiguousarray(block_table, np.int32)
    ctx = np.ascontiguousarray(context_lens, np.int32)
    R = table.shape[0]
    gor = np.zeros(max(R, 1), np.int32)
    gstart = np.zeros(R + 1, np.int32)
    members = np.zeros(max(R, 1), np.int32)
    gblocks = np.zeros(max(R, 1), np.int32)
    cnt = np.zeros(3, np.int32)
    _check(load().pkv_prefix_groups_build(
        _np_ptr(table), table.shape[1], R, _np_ptr(ctx), int(min_shared_blocks), _np_ptr(gor),
        _np_ptr(gstart), _np_ptr(members), _np_ptr(gblocks), _np_ptr(cnt[0:]), _np_ptr(cnt[1:]),
        _np_ptr(cnt[2:])))
    G = int(cnt[0])
    return dict(group_of_req=gor[:R], group_start=gstart[:G + 1], member_req=members[:int(gstart[G])],
                group_blocks=gblocks[:G], num_groups=G, max_group_blocks=int(cnt[1]),
                max_group_members=int(cnt[2]))


# ---- multi-adapter dispatch (host) -------------------------------------------

def pkv_lora_dispatch(adapter_id, prompt_len, bucket_edges=(), max_batch: int = 0):
    """Batches of a multi-adapter request: (order, batches) with order[k] the
    request index of the k-th item executed and batches a list of
    (adapter_id, bucket, start, stop) over order."""
    a = np.ascontiguousarray(adapter_id, np.int32)
    n_ = np.ascontiguousarray(prompt_len, np.int32)
    e = np.ascontiguousarray(bucket_edges, np.int32)
    if a.shape != n_.shape or a.ndim != 1:
        raise ValueError("one adapter id and one prompt length per item")
    n = len(a)
    order = np.zeros(max(n, 1), np.int32)
    start = np.zeros(n + 1, np.int32)
    adp = np.zeros(max(n, 1), np.int32)
    bkt = np.zeros(max(n, 1), np.int32)
    nb = np.zeros(1, np.int32)
    _check(load().pkv_lora_dispatch(_np_ptr(a), _np_ptr(n_), n, _np_ptr(e) if len(e) else None,
                                    len(e), int(max_batch), _np_ptr(order), _np_ptr(start),
                                    _np_ptr(adp), _np_ptr(bkt), _np_ptr(nb)))
    k = int(nb[0])
    return order[:n].tolist(), [(int(adp[b]), int(bkt[b]), int(start[b]), int(start[b + 1]))
                                for b in range(k)]


def pkv_selftest_wait_timeout(pool, limit_us: int = 1000, stream=None):
    """Test aid: one bounded device wait runs out and latches DEVICE_TIMEOUT."""
    _check(load().pkv_selftest_wait_timeout(pool, int(limit_us), _stream(stream)))


def pkv_trace_enable(pool, enable: bool = True):
    _check(load().pkv_trace_enable(pool, 1 if enable else 0))


def pkv_trace_read(pool) -> dict:
    """{kernel name: (launches, total_ms)} since the previous read."""
    arr = (KernelTime * 8)()
    n = np.zeros(1, np.int32)
    _check(load().pkv_trace_read(pool, ctypes.cast(arr, ctypes.c_void_p), 8, _np_ptr(n)))
    return {arr[i].name.decode(): (int(arr[i].launches), float(arr[i].total_ms))
            for i in range(int(n[0]))}


def pkv_check_device_errors(pool, stream=None) -> int:
    out = np.zeros(1, np.int32)
    _check(load().pkv_check_device_errors(pool, _stream(stream), _np_ptr(out)))
    return int(out[0])


def pkv_last_error() -> str:
    return load().pkv_last_error().decode()
