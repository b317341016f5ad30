"""ctypes front end of the fp64 oracle (``pkv_oracle.c``).

TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU baseline).  All arrays are
numpy; bf16 values travel as their uint16 bit patterns and are widened to
float64 exactly inside the C code.
"""

from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pkv_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle_pkv.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (portable C, no target-specific flags)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        lib.oracle_cache_write.argtypes = [P, P, i64, i32, i32, i32, P, P, P, i64]
        lib.oracle_cache_write.restype = i64
        lib.oracle_slot_mapping.argtypes = [P, i32, P, P, i32, i32, P]
        lib.oracle_slot_mapping.restype = i64
        lib.oracle_gather.argtypes = [P, i64, i32, i32, i32, P, i32, P]
        lib.oracle_gather.restype = ctypes.c_int
        lib.oracle_attention.argtypes = [P, P, P, i32, i32, i32, i32, i32, f64, P, P, i32]
        lib.oracle_attention.restype = ctypes.c_int
        lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.oracle_bf16_to_double.restype = f64
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def bf16_to_f64(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def cache_write(k_pool: np.ndarray, v_pool: np.ndarray, k_new: np.ndarray,
                v_new: np.ndarray, slots: np.ndarray) -> int:
    """In-place scatter of new K/V rows into pools shaped [nb][Hkv][B][d]."""
    assert k_pool.flags.c_contiguous and v_pool.flags.c_contiguous
    nb, hkv, bs, d = k_pool.shape
    k_new = _c(k_new, np.uint16)
    v_new = _c(v_new, np.uint16)
    slots = _c(slots, np.int64)
    n = _load().oracle_cache_write(_ptr(k_pool), _ptr(v_pool), nb, hkv, bs, d,
                                   _ptr(k_new), _ptr(v_new), _ptr(slots), len(slots))
    if n < 0:
        raise ValueError("slot outside the pool")
    return int(n)


def slot_mapping(table: np.ndarray, context_lens, new_lens, block_size: int) -> np.ndarray:
    table = _c(table, np.int32)
    ctx = _c(context_lens, np.int32)
    new = _c(new_lens, np.int32)
    out = np.empty(int(new.sum()), np.int64)
    n = _load().oracle_slot_mapping(_ptr(table), table.shape[1], _ptr(ctx), _ptr(new),
                                    len(ctx), block_size, _ptr(out))
    if n < 0:
        raise ValueError("negative table entry inside a context")
    return out


def gather(pool: np.ndarray, table_row, context_len: int) -> np.ndarray:
    """Contiguous [L][Hkv][d] bits of one request's keys or values."""
    nb, hkv, bs, d = pool.shape
    row = _c(table_row, np.int32)
    out = np.empty((context_len, hkv, d), np.uint16)
    rc = _load().oracle_gather(_ptr(_c(pool, np.uint16)), nb, hkv, bs, d, _ptr(row),
                               int(context_len), _ptr(out))
    if rc != 0:
        raise ValueError("bad block-table entry")
    return out


def attention(q_bits: np.ndarray, k_bits: np.ndarray, v_bits: np.ndarray,
              scale: float, threads: int = 1):
    """fp64 attention of one request.

    q_bits [S][Hq][d], k_bits/v_bits [L][Hkv][d] (bf16 bit patterns).  Query i
    sits at absolute position L - S + i and attends to keys 0 .. L - S + i.
    Returns (out [S][Hq][d] float64, lse [S][Hq] float64, natural log).
    """
    q = _c(q_bits, np.uint16)
    k = _c(k_bits, np.uint16)
    v = _c(v_bits, np.uint16)
    S, Hq, d = q.shape
    L, Hkv, d2 = k.shape
    assert d == d2 and v.shape == k.shape
    out = np.zeros((S, Hq, d), np.float64)
    lse = np.zeros((S, Hq), np.float64)
    rc = _load().oracle_attention(_ptr(q), _ptr(k), _ptr(v), S, L, Hq, Hkv, d,
                                  float(scale), _ptr(out), _ptr(lse), int(threads))
    if rc != 0:
        raise ValueError("bad attention shapes")
    return out, lse


def _bits(t) -> np.ndarray:
    """uint16 bit patterns of a bf16 torch tensor (no arithmetic)."""
    import torch
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def request_attention(workload, r: int, threads: int = 1, rows=None):
    """Oracle output of request r of a workload, from its logical K/V.

    ``rows`` (optional) selects query rows: row i is computed alone as a
    single query over keys 0 .. cached+i, which is what it attends to inside
    the full request.
    """
    k, v = workload.request_kv(r)
    q = workload.request_q(r)
    kb, vb, qb = _bits(k), _bits(v), _bits(q)
    if rows is None:
        return attention(qb, kb, vb, workload.scale, threads)
    outs, lses = [], []
    cached = int(workload.cached_lens[r])
    for i in rows:
        L = cached + int(i) + 1
        o, s = attention(qb[i:i + 1], kb[:L], vb[:L], workload.scale, threads)
        outs.append(o[0])
        lses.append(s[0])
    return np.stack(outs), np.stack(lses)


def paged_request_attention(k_pool, v_pool, table_row, context_len: int, q_bits,
                            scale: float, threads: int = 1):
    """Attention of one request read through its block-table row."""
    k = gather(k_pool, table_row, context_len)
    v = gather(v_pool, table_row, context_len)
    return attention(q_bits, k, v, scale, threads)
