"""Thin Python binding of libkvshot's C ABI (include/kvshot.h).

Argument marshalling only: every step of draft attention, draft append and
the gated-delta fusion runs in the library's CUDA kernels.  Tensors are torch CUDA tensors (or raw
device pointers as ints); the current torch stream is used unless a stream
is given.  If the shared library is missing this module raises on import of
the library -- there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import build as _build

KVSHOT_OK = 0
KVSHOT_ERR_NULL = 1
KVSHOT_ERR_SHAPE = 2
KVSHOT_ERR_ALIGN = 3
KVSHOT_ERR_UNSUPPORTED = 4
KVSHOT_ERR_TREE = 5
KVSHOT_ERR_WORKSPACE = 6
KVSHOT_ERR_CUDA = 7
KVSHOT_ERR_DEVICE_BOUNDS = 8
KVSHOT_ERR_TIMEOUT = 9

KVSHOT_TREE = 0x1
KVSHOT_FORCE_CC = 0x2
KVSHOT_FORCE_MMA = 0x4
KVSHOT_FORCE_TC = 0x8
KVSHOT_OVERLAP_PREVIOUS = 0x10
KVSHOT_TARGET_FP8 = 0x20

EXPORTS = ("kvshot_draft_attn", "kvshot_draft_attn_workspace_size", "kvshot_draft_append", "kvshot_status_string",
           "kvshot_version", "kvshot_draft_attn_static", "kvshot_gated_delta", "kvshot_gated_delta_workspace_size",
           "kvshot_kv_project", "kvshot_kv_project_workspace_size", "kvshot_draft_append_qknorm")
KVSHOT_PROJECT_ROPE = 0x1
STATIC_WORKSPACE_BYTES = 64 * 1024 * 1024  # KVSHOT_STATIC_WORKSPACE_BYTES


class KvshotError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: status {status} ({status_string(status)})")
        self.status = status


class AttnDesc(ctypes.Structure):
    """Mirror of kvshot_attn_desc."""

    _fields_ = [
        ("num_caches", ctypes.c_int32),
        ("num_seqs", ctypes.c_int32),
        ("hq", ctypes.c_int32),
        ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("l_cap", ctypes.c_int32),
        ("max_seq_len", ctypes.c_int32),
        ("n_nodes", ctypes.c_int32),
        ("n_query", ctypes.c_int32),
        ("n_max", ctypes.c_int32),
        ("scale", ctypes.c_float),
        ("flags", ctypes.c_uint32),
        ("num_ctas", ctypes.c_int32),
        ("workspace", ctypes.c_void_p),
        ("workspace_bytes", ctypes.c_size_t),
        ("err_flag", ctypes.c_void_p),
        ("k_scale_exp", ctypes.c_int32),
        ("v_scale_exp", ctypes.c_int32),
        ("wait_limit_ns", ctypes.c_uint32),
    ]


class FusionDesc(ctypes.Structure):
    """Mirror of kvshot_fusion_desc."""

    _fields_ = [
        ("num_tokens", ctypes.c_int32),
        ("hidden", ctypes.c_int32),
        ("workspace", ctypes.c_void_p),
        ("workspace_bytes", ctypes.c_size_t),
        ("err_flag", ctypes.c_void_p),
    ]


class ProjectDesc(ctypes.Structure):
    """Mirror of kvshot_project_desc."""

    _fields_ = [
        ("num_tokens", ctypes.c_int32),
        ("num_layers", ctypes.c_int32),
        ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("num_caches", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("l_cap", ctypes.c_int32),
        ("rope_base", ctypes.c_float),
        ("flags", ctypes.c_uint32),
        ("workspace", ctypes.c_void_p),
        ("workspace_bytes", ctypes.c_size_t),
        ("err_flag", ctypes.c_void_p),
    ]


_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libkvshot.so (building it first if requested and needed)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if build_if_missing and not _build.up_to_date():
        _build.build()
    if not os.path.exists(path):
        raise RuntimeError(f"libkvshot.so not found at {path}; run paper_2604_26412_gb300.build.build()")
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    lib.kvshot_draft_attn.argtypes = [ctypes.POINTER(AttnDesc), P, P, P, P, P, P, P, P, P, P, P]
    lib.kvshot_draft_attn.restype = ctypes.c_int
    lib.kvshot_draft_attn_static.argtypes = [ctypes.POINTER(AttnDesc), P, P, P, P, P, P, P, P, P, P, P]
    lib.kvshot_draft_attn_static.restype = ctypes.c_int
    lib.kvshot_draft_attn_workspace_size.argtypes = [ctypes.POINTER(AttnDesc)]
    lib.kvshot_draft_attn_workspace_size.restype = ctypes.c_size_t
    lib.kvshot_draft_append.argtypes = [ctypes.POINTER(AttnDesc), P, P, P, P, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_float, P, P, P, P]
    lib.kvshot_draft_append.restype = ctypes.c_int
    lib.kvshot_draft_append_qknorm.argtypes = [ctypes.POINTER(AttnDesc), P, P, P, P, ctypes.c_int32, ctypes.c_int32,
                                               ctypes.c_float, P, P, ctypes.c_float, P, P, P, P]
    lib.kvshot_draft_append_qknorm.restype = ctypes.c_int
    lib.kvshot_gated_delta.argtypes = [ctypes.POINTER(FusionDesc), P, P, P, P, P, P, P]
    lib.kvshot_gated_delta.restype = ctypes.c_int
    lib.kvshot_gated_delta_workspace_size.argtypes = [ctypes.POINTER(FusionDesc)]
    lib.kvshot_gated_delta_workspace_size.restype = ctypes.c_size_t
    lib.kvshot_kv_project.argtypes = [ctypes.POINTER(ProjectDesc), P, P, P, P, P, P, P, P, P, P]
    lib.kvshot_kv_project.restype = ctypes.c_int
    lib.kvshot_kv_project_workspace_size.argtypes = [ctypes.POINTER(ProjectDesc)]
    lib.kvshot_kv_project_workspace_size.restype = ctypes.c_size_t
    lib.kvshot_status_string.argtypes = [ctypes.c_int]
    lib.kvshot_status_string.restype = ctypes.c_char_p
    lib.kvshot_version.argtypes = []
    lib.kvshot_version.restype = ctypes.c_int32
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().kvshot_status_string(int(status)).decode()


def version() -> int:
    return int(load().kvshot_version())


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, torch.Tensor):
        return x.data_ptr()
    raise TypeError(f"expected a tensor, a device pointer or None, got {type(x)}")


def _dref(desc):
    return None if desc is None else ctypes.byref(desc)


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def make_desc(*, num_caches, num_seqs, hq, hkv, n_nodes, n_query, n_max, max_seq_len, head_dim=128, page_size=0,
              max_pages_per_seq=0, num_pages=0, l_cap=0, scale=0.0, tree=False, flags=0, num_ctas=0,
              workspace=None, workspace_bytes=0, err_flag=None, k_scale_exp=0, v_scale_exp=0,
              wait_limit_ns=0) -> AttnDesc:
    f = int(flags) | (KVSHOT_TREE if tree else 0)
    return AttnDesc(num_caches, num_seqs, hq, hkv, head_dim, page_size, max_pages_per_seq, num_pages, l_cap,
                    max_seq_len, n_nodes, n_query, n_max, float(scale), f, num_ctas, _ptr(workspace),
                    int(workspace_bytes), _ptr(err_flag), int(k_scale_exp), int(v_scale_exp), int(wait_limit_ns))


def workspace_size(desc: AttnDesc) -> int:
    return int(load().kvshot_draft_attn_workspace_size(_dref(desc)))


def draft_attn_status(desc: AttnDesc, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v, tree_parent, out,
                      lse, stream=None) -> int:
    """Call kvshot_draft_attn and return its status code."""
    return int(load().kvshot_draft_attn(_dref(desc), _ptr(q), _ptr(target_k), _ptr(target_v),
                                        _ptr(page_table), _ptr(seq_lens), _ptr(draft_k), _ptr(draft_v),
                                        _ptr(tree_parent), _ptr(out), _ptr(lse), _stream(stream)))


def draft_attn(desc: AttnDesc, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v, tree_parent, out, lse,
               stream=None) -> None:
    st = draft_attn_status(desc, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v, tree_parent, out,
                           lse, stream)
    if st != KVSHOT_OK:
        raise KvshotError(st, "kvshot_draft_attn")


def draft_attn_static_status(desc: AttnDesc, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v,
                             tree_parent, out, lse, stream=None) -> int:
    """Call kvshot_draft_attn_static (library-owned scratch, no allocation) and return its status."""
    return int(load().kvshot_draft_attn_static(_dref(desc), _ptr(q), _ptr(target_k), _ptr(target_v),
                                               _ptr(page_table), _ptr(seq_lens), _ptr(draft_k), _ptr(draft_v),
                                               _ptr(tree_parent), _ptr(out), _ptr(lse), _stream(stream)))


def draft_append_status(desc: AttnDesc, q_in, k_in, v_in, positions, n0: int, n_new: int, rope_base: float, draft_k,
                        draft_v, q_out, stream=None) -> int:
    return int(load().kvshot_draft_append(_dref(desc), _ptr(q_in), _ptr(k_in), _ptr(v_in), _ptr(positions),
                                          int(n0), int(n_new), float(rope_base), _ptr(draft_k), _ptr(draft_v),
                                          _ptr(q_out), _stream(stream)))


def draft_append(desc: AttnDesc, q_in, k_in, v_in, positions, n0: int, n_new: int, rope_base: float, draft_k, draft_v,
                 q_out, stream=None) -> None:
    st = draft_append_status(desc, q_in, k_in, v_in, positions, n0, n_new, rope_base, draft_k, draft_v, q_out, stream)
    if st != KVSHOT_OK:
        raise KvshotError(st, "kvshot_draft_append")


def make_fusion_desc(*, num_tokens, hidden, workspace=None, workspace_bytes=0, err_flag=None) -> FusionDesc:
    return FusionDesc(int(num_tokens), int(hidden), _ptr(workspace), int(workspace_bytes), _ptr(err_flag))


def gated_delta_workspace_size(desc: FusionDesc) -> int:
    return int(load().kvshot_gated_delta_workspace_size(_dref(desc)))


def gated_delta_status(desc: FusionDesc, n, o, w_g, b_g, w_delta, h, stream=None) -> int:
    """Call kvshot_gated_delta (h = n + sigmoid(W_g [n; o; o - n] + b_g) * W_delta (o - n)); return its status."""
    return int(load().kvshot_gated_delta(_dref(desc), _ptr(n), _ptr(o), _ptr(w_g), _ptr(b_g), _ptr(w_delta),
                                         _ptr(h), _stream(stream)))


def gated_delta(desc: FusionDesc, n, o, w_g, b_g, w_delta, h, stream=None) -> None:
    st = gated_delta_status(desc, n, o, w_g, b_g, w_delta, h, stream)
    if st != KVSHOT_OK:
        raise KvshotError(st, "kvshot_gated_delta")


def make_project_desc(*, num_tokens, num_layers, hkv, num_caches, head_dim=128, page_size=0, max_pages_per_seq=0,
                      num_pages=0, l_cap=0, rope_base=1.0e6, rope=True, workspace=None, workspace_bytes=0,
                      err_flag=None) -> ProjectDesc:
    return ProjectDesc(int(num_tokens), int(num_layers), int(hkv), int(head_dim), int(num_caches), int(page_size),
                       int(max_pages_per_seq), int(num_pages), int(l_cap), float(rope_base),
                       KVSHOT_PROJECT_ROPE if rope else 0, _ptr(workspace), int(workspace_bytes), _ptr(err_flag))


def kv_project_workspace_size(desc: ProjectDesc) -> int:
    return int(load().kvshot_kv_project_workspace_size(_dref(desc)))


def kv_project_status(desc: ProjectDesc, k_in, v_in, w_k, w_v, token_cache, positions, page_table, k_out, v_out,
                      stream=None) -> int:
    """Call kvshot_kv_project (K' = W_K [K_1..K_L] (+ RoPE), V' = W_V [V_1..V_L] into the reused cache)."""
    return int(load().kvshot_kv_project(_dref(desc), _ptr(k_in), _ptr(v_in), _ptr(w_k), _ptr(w_v), _ptr(token_cache),
                                        _ptr(positions), _ptr(page_table), _ptr(k_out), _ptr(v_out), _stream(stream)))


def kv_project(desc: ProjectDesc, k_in, v_in, w_k, w_v, token_cache, positions, page_table, k_out, v_out,
               stream=None) -> None:
    st = kv_project_status(desc, k_in, v_in, w_k, w_v, token_cache, positions, page_table, k_out, v_out, stream)
    if st != KVSHOT_OK:
        raise KvshotError(st, "kvshot_kv_project")


def draft_append_qknorm_status(desc: AttnDesc, q_in, k_in, v_in, positions, n0: int, n_new: int, rope_base: float,
                               q_norm_w, k_norm_w, eps: float, draft_k, draft_v, q_out, stream=None) -> int:
    return int(load().kvshot_draft_append_qknorm(_dref(desc), _ptr(q_in), _ptr(k_in), _ptr(v_in), _ptr(positions),
                                                 int(n0), int(n_new), float(rope_base), _ptr(q_norm_w),
                                                 _ptr(k_norm_w), float(eps), _ptr(draft_k), _ptr(draft_v),
                                                 _ptr(q_out), _stream(stream)))


def draft_append_qknorm(desc: AttnDesc, q_in, k_in, v_in, positions, n0: int, n_new: int, rope_base: float, q_norm_w,
                        k_norm_w, eps: float, draft_k, draft_v, q_out, stream=None) -> None:
    st = draft_append_qknorm_status(desc, q_in, k_in, v_in, positions, n0, n_new, rope_base, q_norm_w, k_norm_w, eps,
                                    draft_k, draft_v, q_out, stream)
    if st != KVSHOT_OK:
        raise KvshotError(st, "kvshot_draft_append_qknorm")
