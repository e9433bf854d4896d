"""ctypes declarations of the C ABI in include/shallowstream.h (marshalling only)."""
from __future__ import annotations

import ctypes as C
import os

from . import build as _build

c_status = C.c_int


class IndexConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("n_q_heads", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("tokens_per_frame", C.c_int32),
                ("frames_per_unit", C.c_int32), ("max_frames", C.c_int64)]


ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p)
FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p, C.c_void_p)


class Allocator(C.Structure):
    _fields_ = [("alloc", ALLOC_FN), ("free", FREE_FN), ("ctx", C.c_void_p)]


class IndexView(C.Structure):
    _fields_ = [("n_frames", C.c_int64), ("n_units", C.c_int64), ("token_capacity", C.c_int64),
                ("keys", C.c_void_p), ("descriptors", C.c_void_p), ("n_windows", C.c_int32),
                ("window_frames", C.c_int32), ("n_centroids", C.c_int32),
                ("centroids", C.c_void_p), ("assignment", C.c_void_p),
                ("window_first_unit", C.c_void_p), ("member_counts", C.c_void_p),
                ("member_sizes", C.c_void_p), ("n_clustered_units", C.c_int64),
                ("cluster_capacity", C.c_int32), ("unit_cluster", C.c_void_p),
                ("cluster_count", C.c_void_p), ("cluster_centroids", C.c_void_p),
                ("cluster_sizes", C.c_void_p), ("cluster_keys", C.c_void_p),
                ("values", C.c_void_p), ("n_value_frames", C.c_int64)]


class CompressParams(C.Structure):
    _fields_ = [("window_frames", C.c_int32), ("n_centroids", C.c_int32), ("iters", C.c_int32),
                ("first_frame", C.c_int64), ("n_frames", C.c_int64)]


class RetrieveParams(C.Structure):
    _fields_ = [("k", C.c_int32), ("budget_units", C.c_int32), ("pool_mult", C.c_int32),
                ("n_prev", C.c_int32), ("n_recent_units", C.c_int32), ("q_agg", C.c_int32),
                ("head_agg", C.c_int32), ("use_clusters", C.c_int32)]


class Result(C.Structure):
    _fields_ = [("topk_tok", C.c_void_p), ("topk_w", C.c_void_p), ("list_stats", C.c_void_p),
                ("unit_votes", C.c_void_p), ("unit_mass", C.c_void_p), ("pool", C.c_void_p),
                ("sel_units", C.c_void_p), ("exp_units", C.c_void_p), ("frames", C.c_void_p),
                ("counts", C.c_void_p), ("status", C.c_void_p)]


class HostResult(C.Structure):
    _fields_ = [("sel_units", C.c_void_p), ("exp_units", C.c_void_p), ("frames", C.c_void_p),
                ("counts", C.c_void_p)]


class ShardResult(C.Structure):
    _fields_ = [("topk_tok", C.c_void_p), ("topk_s", C.c_void_p), ("list_stats", C.c_void_p),
                ("unit_stats", C.c_void_p), ("status", C.c_void_p)]


class Shard(C.Structure):
    _fields_ = [("unit_begin", C.c_int64), ("n_units", C.c_int32), ("topk_tok", C.c_void_p),
                ("topk_s", C.c_void_p), ("list_stats", C.c_void_p),
                ("unit_stats", C.c_void_p), ("desc", C.c_void_p)]


class MergeResult(C.Structure):
    _fields_ = [("topk_tok", C.c_void_p), ("topk_w", C.c_void_p), ("list_stats", C.c_void_p),
                ("unit_votes", C.c_void_p), ("unit_mass", C.c_void_p), ("pool", C.c_void_p),
                ("sel_units", C.c_void_p), ("exp_units", C.c_void_p), ("frames", C.c_void_p),
                ("counts", C.c_void_p)]


class ForwardParams(C.Structure):
    _fields_ = [("intermediate", C.c_int32), ("rms_eps", C.c_float), ("rope_theta", C.c_float),
                ("pos0", C.c_int64)]


class LayerWeights(C.Structure):
    _fields_ = [("ln1", C.c_void_p), ("wqkv", C.c_void_p), ("bqkv", C.c_void_p),
                ("wo", C.c_void_p), ("ln2", C.c_void_p), ("wgu", C.c_void_p), ("wd", C.c_void_p)]


class Trace(C.Structure):
    _fields_ = [("score_begin", C.c_void_p), ("score_end", C.c_void_p)]


# name -> (restype, argtypes); every entry point declared in include/shallowstream.h
SIGNATURES = {
    "ss_status_string": (C.c_char_p, [c_status]),
    "ss_last_error": (C.c_char_p, []),
    "ss_version": (C.c_char_p, []),
    "ss_index_create": (c_status, [C.POINTER(IndexConfig), C.POINTER(Allocator), C.c_void_p,
                                   C.POINTER(C.c_void_p)]),
    "ss_index_destroy": (c_status, [C.c_void_p]),
    "ss_index_append": (c_status, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int64, C.c_void_p]),
    "ss_index_get_view": (c_status, [C.c_void_p, C.POINTER(IndexView)]),
    "ss_index_compress": (c_status, [C.c_void_p, C.POINTER(CompressParams), C.c_void_p]),
    "ss_retrieve_workspace_size": (c_status, [C.POINTER(C.c_void_p), C.c_int32,
                                              C.POINTER(C.c_int32), C.POINTER(RetrieveParams),
                                              C.POINTER(C.c_size_t)]),
    "ss_retrieve": (c_status, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(RetrieveParams),
                               C.POINTER(Result), C.c_void_p, C.c_size_t, C.c_void_p,
                               C.POINTER(Trace)]),
    "ss_retrieve_batched": (c_status, [C.POINTER(C.c_void_p), C.POINTER(C.c_void_p),
                                       C.POINTER(C.c_int32), C.c_int32,
                                       C.POINTER(RetrieveParams), C.POINTER(Result),
                                       C.c_void_p, C.c_size_t, C.c_void_p, C.POINTER(Trace)]),
    "ss_retrieve_host": (c_status, [C.c_void_p, C.c_void_p, C.c_int32,
                                    C.POINTER(RetrieveParams), C.POINTER(HostResult),
                                    C.c_void_p, C.c_size_t, C.c_void_p]),
    "ss_retrieve_static": (c_status, [C.c_void_p, C.c_void_p, C.c_int32,
                                      C.POINTER(RetrieveParams), C.POINTER(Result),
                                      C.c_void_p]),
    "ss_status_sync": (c_status, [C.c_void_p, C.c_void_p]),
    "ss_set_wait_limit": (c_status, [C.c_int64]),
    "ss_retrieve_shard": (c_status, [C.c_void_p, C.c_void_p, C.c_int32,
                                     C.POINTER(RetrieveParams), C.c_int64,
                                     C.POINTER(ShardResult), C.c_void_p, C.c_size_t,
                                     C.c_void_p]),
    "ss_index_cluster_units": (c_status, [C.c_void_p, C.c_int64, C.c_float, C.c_int32,
                                          C.c_void_p]),
    "ss_index_units_over_budget": (c_status, [C.c_void_p, C.c_int64, C.c_int64,
                                              C.POINTER(C.c_int64)]),
    "ss_select_clusters": (c_status, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                      C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "ss_index_get_config": (c_status, [C.c_void_p, C.POINTER(IndexConfig)]),
    "ss_index_save": (c_status, [C.c_void_p, C.c_char_p, C.c_void_p]),
    "ss_index_load": (c_status, [C.c_char_p, C.POINTER(Allocator), C.c_void_p,
                                 C.POINTER(C.c_void_p)]),
    "ss_index_append_values": (c_status, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int64,
                                          C.c_void_p]),
    "ss_forward_workspace_size": (c_status, [C.c_void_p, C.c_int32, C.POINTER(ForwardParams),
                                             C.POINTER(C.c_size_t)]),
    "ss_question_forward": (c_status, [C.c_void_p, C.POINTER(LayerWeights),
                                       C.POINTER(ForwardParams), C.c_void_p, C.c_int32,
                                       C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                       C.c_size_t, C.c_void_p]),
    "ss_merge_shards": (c_status, [C.POINTER(Shard), C.c_int32, C.c_int32, C.c_int32,
                                   C.c_int32, C.c_int32, C.POINTER(RetrieveParams),
                                   C.POINTER(MergeResult)]),
}

_LIB = None


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None) -> C.CDLL:
    """Loads the built library (raises if it has not been built)."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    p = path or os.environ.get("SHALLOWSTREAM_LIB") or _build.LIB
    if not os.path.exists(p):
        raise RuntimeError(f"CUDA library not built ({p} missing): run "
                           "paper_2609_02780_gb300.build.build() or __graft_entry__.build()")
    lib = C.CDLL(p)
    for name, (res, args) in SIGNATURES.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    if path is None:
        _LIB = lib
    return lib
