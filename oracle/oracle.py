"""CPU fp64 oracle for KV-reuse draft attention -- numpy front end.

TEST INFRASTRUCTURE ONLY.  This module and the C++ code it loads are the
plain definition the CUDA library is checked against.  Only tests, the
package's ``smoke()`` self-check and ``bench.py``'s CPU-baseline leg may import
it; the library itself never does, and nothing here imports the library.

Definitions (cited from the paper, arXiv 2604.26412):
  * attention over the memory M_i: Sec. 2.2 Eq. "kv-reattention" and Sec. 3.4
    Eq. "cross-attn" / App. B "Cross-attention memory" -- verified prefix tokens
    use the target model's K/V, draft positions use the drafter's own K/V;
  * the chain / tree ancestor mask of speculative drafting (Sec. 3.5 tree
    (8, 10, 60)); a node sees itself and its ancestors;
  * RoPE re-application to drafted keys (Sec. 3.2, "Proj + RoPE fix").

Inputs are numpy arrays: bf16 tensors as uint16 bit patterns, int32 metadata.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libkvshot_oracle.so")
_SRC = os.path.join(_HERE, "kvshot_oracle.cpp")
_HDR = os.path.join(_HERE, "kvshot_oracle.h")
_lock = threading.Lock()
_lib = None

ERR_SHAPE = 2
ERR_TREE = 5
ERR_PAGE = 8


class OracleError(RuntimeError):
    pass


class KvoDesc(ctypes.Structure):
    _fields_ = [
        ("num_caches", ctypes.c_int32),
        ("num_seqs", ctypes.c_int32),
        ("hq", ctypes.c_int32),
        ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("paged", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("l_cap", ctypes.c_int32),
        ("n_nodes", ctypes.c_int32),
        ("n_query", ctypes.c_int32),
        ("n_max", ctypes.c_int32),
        ("tree", ctypes.c_int32),
        ("scale", ctypes.c_double),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (plain -O2, portable flags) into oracle/_build."""
    with _lock:
        newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
        if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= newest:
            return _LIB_PATH
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread", "-o", tmp, _SRC]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        # KVO_LIB_OVERRIDE loads a deliberately altered oracle build (used by the
        # test that checks the pins catch planted mistakes).
        path = os.environ.get("KVO_LIB_OVERRIDE") or build()
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        lib.kvo_attn.argtypes = [ctypes.POINTER(KvoDesc), P, P, P, P, P, P, P, P, P, P, ctypes.c_int]
        lib.kvo_attn.restype = ctypes.c_int
        lib.kvo_attn_probs.argtypes = [ctypes.POINTER(KvoDesc), P, P, P, P, P, P,
                                       ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, P]
        lib.kvo_attn_probs.restype = ctypes.c_int
        lib.kvo_append.argtypes = [ctypes.POINTER(KvoDesc), P, P, P, P, ctypes.c_int32, ctypes.c_int32,
                                   ctypes.c_double, P, P, P, P, P]
        lib.kvo_append.restype = ctypes.c_int
        lib.kvo_round_bf16.argtypes = [ctypes.c_double]
        lib.kvo_round_bf16.restype = ctypes.c_uint16
        _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError(f"bf16 arrays are passed as uint16 bit patterns, got {a.dtype}")
    return a


def _i32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.int32)


def make_desc(*, num_caches, num_seqs, hq, hkv, head_dim, n_nodes, n_query, n_max, tree,
              paged=False, page_size=0, max_pages_per_seq=0, num_pages=0, l_cap=0, scale=0.0):
    return KvoDesc(num_caches, num_seqs, hq, hkv, head_dim, int(paged), page_size, max_pages_per_seq,
                   num_pages, l_cap, n_nodes, n_query, n_max, int(tree), float(scale))


def attn(desc: KvoDesc, q, tk, tv, page_table, seq_lens, dk, dv, tree_parent, nthreads: int = 0):
    """Return (out [C, Nq, hq, D] float64, lse [C, Nq, hq] float64)."""
    lib = _load()
    q, tk, tv, dk, dv = map(_u16, (q, tk, tv, dk, dv))
    page_table, seq_lens, tree_parent = map(_i32, (page_table, seq_lens, tree_parent))
    out = np.empty((desc.num_caches, desc.n_query, desc.hq, desc.head_dim), np.float64)
    lse = np.empty((desc.num_caches, desc.n_query, desc.hq), np.float64)
    rc = lib.kvo_attn(ctypes.byref(desc), _ptr(q), _ptr(tk), _ptr(tv), _ptr(page_table), _ptr(seq_lens),
                      _ptr(dk), _ptr(dv), _ptr(tree_parent), _ptr(out), _ptr(lse), int(nthreads))
    if rc:
        raise OracleError(f"kvo_attn failed with code {rc}")
    return out, lse


def attn_probs(desc: KvoDesc, q, tk, page_table, seq_lens, dk, tree_parent, c, n_local, h):
    """Probabilities of one query row over [prefix keys 0..L_c) + [draft slots 0..N)."""
    lib = _load()
    q, tk, dk = map(_u16, (q, tk, dk))
    page_table, seq_lens, tree_parent = map(_i32, (page_table, seq_lens, tree_parent))
    probs = np.empty(int(seq_lens[c]) + desc.n_nodes, np.float64)
    rc = lib.kvo_attn_probs(ctypes.byref(desc), _ptr(q), _ptr(tk), _ptr(page_table), _ptr(seq_lens),
                            _ptr(dk), _ptr(tree_parent), int(c), int(n_local), int(h), _ptr(probs))
    if rc:
        raise OracleError(f"kvo_attn_probs failed with code {rc}")
    return probs


def append(desc: KvoDesc, q_in, k_in, v_in, positions, n0, n_new, rope_base, draft_k, draft_v,
           want_f64: bool = False):
    """RoPE + append.  draft_k / draft_v (uint16) are updated in place.

    Returns q_out (uint16 [C, n_new, hq, D]); with want_f64 also the unrounded
    rotated q and k (float64, in the q_in / k_in layouts)."""
    lib = _load()
    q_in, k_in, v_in = map(_u16, (q_in, k_in, v_in))
    positions = _i32(positions)
    for buf in (draft_k, draft_v):
        if buf.dtype != np.uint16 or not buf.flags["C_CONTIGUOUS"]:
            raise TypeError("draft buffers must be C-contiguous uint16 arrays")
    q_out = np.empty(q_in.shape, np.uint16)
    q_rot = np.empty(q_in.shape, np.float64) if want_f64 else None
    k_rot = np.empty(k_in.shape, np.float64) if want_f64 else None
    rc = lib.kvo_append(ctypes.byref(desc), _ptr(q_in), _ptr(k_in), _ptr(v_in), _ptr(positions), int(n0),
                        int(n_new), float(rope_base), _ptr(draft_k), _ptr(draft_v), _ptr(q_out),
                        _ptr(q_rot), _ptr(k_rot))
    if rc:
        raise OracleError(f"kvo_append failed with code {rc}")
    return (q_out, q_rot, k_rot) if want_f64 else q_out


def round_bf16(x: float) -> int:
    return int(_load().kvo_round_bf16(float(x)))
