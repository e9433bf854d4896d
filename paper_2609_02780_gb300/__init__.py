"""GB300-native query-time evidence retrieval over a shallow-layer key index
(ShallowStream, arxiv 2609.02780, Sec. 4.1-4.2).

Thin Python binding of the C ABI in include/shallowstream.h: it marshals torch
tensors (device memory, the current CUDA stream) into the library's calls. Every
step of retrieval runs in the library's CUDA kernels; there is no Python or CPU
fallback, and using the binding without the built library raises.

    idx = Index(n_layers=4, n_q_heads=28, n_kv_heads=4, tokens_per_frame=196,
                max_frames=3600)
    idx.append(keys)                 # bf16 [P][Hkv][n_frames * T_f][128] on the GPU
    r = idx.retrieve(q, k=1024, budget=64)   # q: bf16 [P][R][Hq][128]
    r.frames()                       # selected + expanded frames, ascending
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import torch

from . import _abi

Q_LAST, Q_MEAN_LOGIT, Q_MEAN_SOFTMAX = 0, 1, 2
H_PER_QHEAD, H_MEAN = 0, 1
CENTROID_ID_BASE = 0x40000000
STATUS_NAMES = ("OK", "INVALID_ARG", "UNSUPPORTED", "CAPACITY", "STATE", "ALLOC", "CUDA",
                "TIMEOUT", "INTERNAL")


class ShallowStreamError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"SS_ERR_{name}: {message}" if status else message)


def _lib():
    return _abi.load()


def _check(status: int) -> None:
    if status != 0:
        msg = _lib().ss_last_error().decode(errors="replace")
        raise ShallowStreamError(status, msg)


def _stream_ptr(device: torch.device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


def version() -> str:
    return _lib().ss_version().decode()


@dataclass
class RetrieveParams:
    k: int
    budget: int
    pool_mult: int = 4
    n_prev: int = 1
    n_recent: int = 0
    q_agg: int = Q_LAST
    head_agg: int = H_PER_QHEAD
    use_clusters: int = 0

    def to_c(self) -> _abi.RetrieveParams:
        return _abi.RetrieveParams(self.k, self.budget, self.pool_mult, self.n_prev,
                                   self.n_recent, self.q_agg, self.head_agg,
                                   self.use_clusters)


class Result:
    """Device tensors written by one retrieval (valid once the stream reaches them)."""

    def __init__(self, idx: "Index", p: RetrieveParams):
        dev = idx.device
        n_lists = idx.n_layers * (1 if p.head_agg == H_MEAN else idx.n_q_heads)
        pool = min(p.pool_mult * p.budget, idx.unit_capacity)
        nexp = p.budget * (1 + p.n_prev)
        i32 = dict(dtype=torch.int32, device=dev)
        f32 = dict(dtype=torch.float32, device=dev)
        self.params = p
        self.frames_per_unit = idx.frames_per_unit
        self.topk_tok = torch.empty(n_lists, p.k, **i32)
        self.topk_w = torch.empty(n_lists, p.k, **f32)
        self.list_stats = torch.empty(n_lists, 2, **f32)
        self.unit_votes = torch.empty(idx.unit_capacity, **i32)
        self.unit_mass = torch.empty(idx.unit_capacity, **f32)
        self.pool = torch.empty(pool, **i32)
        self.sel_units = torch.empty(p.budget, **i32)
        self.exp_units = torch.empty(nexp, **i32)
        self.frames_buf = torch.empty(nexp * idx.frames_per_unit, **i32)
        self.counts = torch.empty(4, **i32)
        self.status = torch.empty(1, **i32)

    def to_c(self) -> _abi.Result:
        return _abi.Result(self.topk_tok.data_ptr(), self.topk_w.data_ptr(),
                           self.list_stats.data_ptr(), self.unit_votes.data_ptr(),
                           self.unit_mass.data_ptr(), self.pool.data_ptr(),
                           self.sel_units.data_ptr(), self.exp_units.data_ptr(),
                           self.frames_buf.data_ptr(), self.counts.data_ptr(),
                           self.status.data_ptr())

    def check(self) -> None:
        """Synchronizes the current stream and raises on a device-side error."""
        dev = self.status.device
        _check(_lib().ss_status_sync(C.c_void_p(self.status.data_ptr()),
                                     C.c_void_p(_stream_ptr(dev))))

    def host(self) -> dict:
        """Synchronizes and returns the selection as Python lists."""
        self.check()
        c = self.counts.cpu().tolist()
        return {"pool": self.pool[:c[0]].cpu().tolist(),
                "sel": self.sel_units[:c[1]].cpu().tolist(),
                "expanded": self.exp_units[:c[2]].cpu().tolist(),
                "frames": self.frames_buf[:c[3]].cpu().tolist()}

    def frames(self) -> list[int]:
        return self.host()["frames"]


@dataclass
class ForwardParams:
    """ss_forward_params: MLP width, RMSNorm epsilon, RoPE base, position of row 0
    (< 0: the stored token count)."""
    intermediate: int
    rms_eps: float = 1e-6
    rope_theta: float = 1e6
    pos0: int = -1

    def abi(self) -> _abi.ForwardParams:
        return _abi.ForwardParams(self.intermediate, self.rms_eps, self.rope_theta, self.pos0)


class Index:
    """A shallow key index (Eq. 2) of one video stream, resident on one GPU."""

    def __init__(self, n_layers: int, n_q_heads: int, n_kv_heads: int,
                 tokens_per_frame: int, max_frames: int, frames_per_unit: int = 1,
                 head_dim: int = 128, device=None):
        lib = _lib()
        d = torch.device(device) if device is not None else torch.device("cuda")
        if d.type != "cuda":
            raise ValueError("an index lives on a CUDA device")
        self.device = d if d.index is not None else torch.device("cuda", torch.cuda.current_device())
        self.n_layers, self.n_q_heads, self.n_kv_heads = n_layers, n_q_heads, n_kv_heads
        self.tokens_per_frame, self.frames_per_unit = tokens_per_frame, frames_per_unit
        self.max_frames = max_frames
        self.unit_capacity = max_frames // frames_per_unit
        self._blocks: dict[int, torch.Tensor] = {}
        self._alloc_cb = _abi.ALLOC_FN(self._alloc)
        self._free_cb = _abi.FREE_FN(self._free)
        self._allocator = _abi.Allocator(self._alloc_cb, self._free_cb, None)
        self._ws: torch.Tensor | None = None
        self._host_calls: dict = {}  # retrieve_host: per (rows, params) call state
        cfg = _abi.IndexConfig(n_layers, n_q_heads, n_kv_heads, head_dim, tokens_per_frame,
                               frames_per_unit, max_frames)
        h = C.c_void_p()
        with torch.cuda.device(self.device):
            _check(lib.ss_index_create(C.byref(cfg), C.byref(self._allocator),
                                       C.c_void_p(_stream_ptr(self.device)), C.byref(h)))
        self._h = h

    @classmethod
    def load(cls, path: str, device=None) -> "Index":
        """ss_index_load: an index recreated from a checkpoint file of save()."""
        lib = _lib()
        self = cls.__new__(cls)
        d = torch.device(device) if device is not None else torch.device("cuda")
        self.device = d if d.index is not None else torch.device("cuda", torch.cuda.current_device())
        self._blocks = {}
        self._alloc_cb = _abi.ALLOC_FN(self._alloc)
        self._free_cb = _abi.FREE_FN(self._free)
        self._allocator = _abi.Allocator(self._alloc_cb, self._free_cb, None)
        self._ws = None
        self._host_calls = {}
        self._h = None
        h = C.c_void_p()
        with torch.cuda.device(self.device):
            _check(lib.ss_index_load(str(path).encode(), C.byref(self._allocator),
                                     C.c_void_p(_stream_ptr(self.device)), C.byref(h)))
        self._h = h
        cfg = _abi.IndexConfig()
        _check(lib.ss_index_get_config(h, C.byref(cfg)))
        self.n_layers, self.n_q_heads, self.n_kv_heads = cfg.n_layers, cfg.n_q_heads, cfg.n_kv_heads
        self.tokens_per_frame, self.frames_per_unit = cfg.tokens_per_frame, cfg.frames_per_unit
        self.max_frames = cfg.max_frames
        self.unit_capacity = cfg.max_frames // cfg.frames_per_unit
        return self

    def save(self, path: str) -> None:
        """ss_index_save: writes a checkpoint of the index to `path` (synchronous)."""
        with torch.cuda.device(self.device):
            _check(_lib().ss_index_save(self.handle, str(path).encode(),
                                        C.c_void_p(_stream_ptr(self.device))))

    # allocator callbacks: device memory comes from torch's caching allocator
    def _alloc(self, nbytes, stream, ctx):
        try:
            t = torch.empty(int(nbytes), dtype=torch.uint8, device=self.device)
        except Exception:
            return None
        self._blocks[t.data_ptr()] = t
        return t.data_ptr()

    def _free(self, ptr, stream, ctx):
        self._blocks.pop(ptr, None)

    @property
    def handle(self) -> C.c_void_p:
        if self._h is None:
            raise RuntimeError("index destroyed")
        return self._h

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            torch.cuda.synchronize(self.device)
            _lib().ss_index_destroy(self._h)
            self._h = None
            self._blocks.clear()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def view(self) -> _abi.IndexView:
        v = _abi.IndexView()
        _check(_lib().ss_index_get_view(self.handle, C.byref(v)))
        return v

    @property
    def n_frames(self) -> int:
        return self.view().n_frames

    @property
    def n_units(self) -> int:
        return self.view().n_units

    def _block_view(self, ptr: int, dtype, shape) -> torch.Tensor:
        t = self._blocks[ptr]
        return t.view(dtype)[: torch.Size(shape).numel()].view(*shape)

    def descriptors(self) -> torch.Tensor:
        """Device fp32 [n_units][Hkv * 128] unit descriptors (Eq. 3), a view."""
        v = self.view()
        d = self._block_view(v.descriptors, torch.float32,
                             (self.unit_capacity, self.n_kv_heads * 128))
        return d[: v.n_units]

    def keys(self) -> torch.Tensor:
        """Device bf16 [P][Hkv][capacity][128] key slabs, a view."""
        v = self.view()
        return self._block_view(v.keys, torch.bfloat16,
                                (self.n_layers, self.n_kv_heads, v.token_capacity, 128))

    def clusters(self) -> dict:
        """Views of the compressed windows' device arrays (after compress()):
        centroids bf16 [P][Hkv][n_windows][n_c][128], assignment uint8 [P][Hkv][capacity],
        member_counts int32 [P][Hkv][n_windows][n_c][units per window], member_sizes
        int32 [P][Hkv][n_windows][n_c], window_first_unit int32 [n_windows]."""
        v = self.view()
        if v.window_frames == 0:
            raise ValueError("the index has no compressed windows")
        P, H, nc = self.n_layers, self.n_kv_heads, v.n_centroids
        wcap = self.unit_capacity * self.frames_per_unit // v.window_frames
        wu = v.window_frames // self.frames_per_unit
        nw = v.n_windows
        cent = self._block_view(v.centroids, torch.bfloat16, (P, H, wcap, nc, 128))
        asg = self._block_view(v.assignment, torch.uint8, (P, H, v.token_capacity))
        mc = self._block_view(v.member_counts, torch.int32, (P, H, wcap, nc, wu))
        ms = self._block_view(v.member_sizes, torch.int32, (P, H, wcap, nc))
        wf = self._block_view(v.window_first_unit, torch.int32, (wcap,))
        return {"centroids": cent[:, :, :nw], "assignment": asg,
                "member_counts": mc[:, :, :nw], "member_sizes": ms[:, :, :nw],
                "window_first_unit": wf[:nw], "window_frames": v.window_frames,
                "n_centroids": nc}

    def cluster_units(self, n_units: int, tau: float, max_clusters: int) -> None:
        """ss_index_cluster_units: the next n_units oldest detailed units leave the detailed
        window and join clusters (Sec. 4.1, Eq. 6-7)."""
        with torch.cuda.device(self.device):
            _check(_lib().ss_index_cluster_units(self.handle, int(n_units), float(tau),
                                                 int(max_clusters),
                                                 C.c_void_p(_stream_ptr(self.device))))

    def units_over_budget(self, budget_bytes: int, near_term_units: int) -> int:
        """ss_index_units_over_budget (Eq. 5): detailed units that must leave."""
        n = C.c_int64()
        _check(_lib().ss_index_units_over_budget(self.handle, int(budget_bytes),
                                                 int(near_term_units), C.byref(n)))
        return n.value

    def unit_clusters(self) -> dict:
        """Views of the long-history compression's device arrays: unit_cluster [n_clustered],
        centroids [C][Hkv * 128], sizes [C], keys fp32 [C][P][Hkv][T_u][128]."""
        v = self.view()
        if v.cluster_capacity == 0:
            raise ValueError("the index has no unit clusters")
        cap = v.cluster_capacity
        tu = self.tokens_per_frame * self.frames_per_unit
        cnt = self._block_view(v.cluster_count, torch.int32, (1,))
        n_c = int(cnt.item())
        uc = self._block_view(v.unit_cluster, torch.int32, (self.unit_capacity,))
        cen = self._block_view(v.cluster_centroids, torch.float32, (cap, self.n_kv_heads * 128))
        sz = self._block_view(v.cluster_sizes, torch.int32, (cap,))
        ck = self._block_view(v.cluster_keys, torch.float32,
                              (cap, self.n_layers, self.n_kv_heads, tu, 128))
        return {"n_clustered_units": v.n_clustered_units, "unit_cluster": uc[:v.n_clustered_units],
                "centroids": cen[:n_c], "sizes": sz[:n_c], "keys": ck[:n_c]}

    def select_clusters(self, q: torch.Tensor, k_l: int, q_agg: int = Q_LAST) -> dict:
        """ss_select_clusters (Eq. 13): the top k_l clusters for question rows q."""
        if q.dtype != torch.bfloat16 or q.dim() != 4 or not q.is_contiguous() or q.device != self.device:
            raise ValueError("q must be contiguous bf16 [P][R][Hq][128] on the index's device")
        ids = torch.empty(k_l, dtype=torch.int32, device=self.device)
        sc = torch.empty(k_l, dtype=torch.float32, device=self.device)
        cnt = torch.empty(1, dtype=torch.int32, device=self.device)
        with torch.cuda.device(self.device):
            _check(_lib().ss_select_clusters(self.handle, C.c_void_p(q.data_ptr()), q.shape[1],
                                             int(q_agg), int(k_l), C.c_void_p(ids.data_ptr()),
                                             C.c_void_p(sc.data_ptr()), C.c_void_p(cnt.data_ptr()),
                                             C.c_void_p(_stream_ptr(self.device))))
        return {"ids": ids, "scores": sc, "count": cnt, "_keep": q}

    def append(self, keys: torch.Tensor, n_frames: int | None = None) -> None:
        """Appends frames of shallow keys bf16 [P][Hkv][S][128] (the first
        n_frames * T_f tokens of each slab; S may exceed that)."""
        if keys.dtype != torch.bfloat16 or keys.dim() != 4:
            raise ValueError("keys must be bf16 [P][Hkv][S][128]")
        if keys.device != self.device:
            raise ValueError("keys must be on the index's device")
        if keys.stride(3) != 1 or keys.stride(2) != 128 or keys.stride(0) != keys.shape[1] * keys.stride(1):
            raise ValueError("keys must be row-major per slab")
        S = keys.stride(1) // 128
        if n_frames is None:
            if keys.shape[2] % self.tokens_per_frame:
                raise ValueError("token count is not a whole number of frames")
            n_frames = keys.shape[2] // self.tokens_per_frame
        with torch.cuda.device(self.device):
            _check(_lib().ss_index_append(self.handle, C.c_void_p(keys.data_ptr()),
                                          int(n_frames), int(S),
                                          C.c_void_p(_stream_ptr(self.device))))
        self._last_src = keys  # keep the source alive until the stream passes the copy

    def append_values(self, values: torch.Tensor, n_frames: int | None = None) -> None:
        """Stores the values bf16 [P][Hkv][S][128] of the next frames whose keys are
        stored (ss_index_append_values; the question's forward reads them)."""
        if values.dtype != torch.bfloat16 or values.dim() != 4 or values.device != self.device:
            raise ValueError("values must be bf16 [P][Hkv][S][128] on the index's device")
        if (values.stride(3) != 1 or values.stride(2) != 128 or
                values.stride(0) != values.shape[1] * values.stride(1)):
            raise ValueError("values must be row-major per slab")
        S = values.stride(1) // 128
        if n_frames is None:
            if values.shape[2] % self.tokens_per_frame:
                raise ValueError("token count is not a whole number of frames")
            n_frames = values.shape[2] // self.tokens_per_frame
        with torch.cuda.device(self.device):
            _check(_lib().ss_index_append_values(self.handle, C.c_void_p(values.data_ptr()),
                                                 int(n_frames), int(S),
                                                 C.c_void_p(_stream_ptr(self.device))))
        self._last_vsrc = values

    def values(self) -> torch.Tensor:
        """Device bf16 [P][Hkv][capacity][128] value slabs, a view."""
        v = self.view()
        if not v.values:
            raise ValueError("the index stores no values")
        return self._block_view(v.values, torch.bfloat16,
                                (self.n_layers, self.n_kv_heads, v.token_capacity, 128))

    def forward_workspace_bytes(self, n_rows: int, params: "ForwardParams") -> int:
        n = C.c_size_t()
        fp = params.abi()
        _check(_lib().ss_forward_workspace_size(self.handle, int(n_rows), C.byref(fp),
                                                C.byref(n)))
        return n.value

    def forward(self, layers: list[dict], h_in: torch.Tensor, params: "ForwardParams", *,
                q_out: torch.Tensor | None = None, h_out: torch.Tensor | None = None,
                status: torch.Tensor | None = None,
                workspace: torch.Tensor | None = None) -> tuple[torch.Tensor, torch.Tensor]:
        """ss_question_forward (Sec. 4.2, Eq. 10): the question's rows h_in bf16 [R][D]
        through the P shallow layers (weights: one dict per layer of bf16 device tensors
        ln1, wqkv, bqkv (or None), wo, ln2, wgu, wd). Returns (q bf16 [P][R][Hq][128], the
        retrieval's input, and H fp32 [R][D]). Asynchronous on the current stream."""
        if len(layers) != self.n_layers:
            raise ValueError("one weight dict per shallow layer")
        D = self.n_q_heads * 128
        if (h_in.dtype != torch.bfloat16 or h_in.dim() != 2 or h_in.shape[1] != D or
                not h_in.is_contiguous() or h_in.device != self.device):
            raise ValueError("h_in must be contiguous bf16 [R][Hq * 128] on the index's device")
        R = h_in.shape[0]
        if q_out is None:
            q_out = torch.empty(self.n_layers, R, self.n_q_heads, 128, dtype=torch.bfloat16,
                                device=self.device)
        if h_out is None:
            h_out = torch.empty(R, D, dtype=torch.float32, device=self.device)
        W = (_abi.LayerWeights * self.n_layers)()
        keep = []
        for i, w in enumerate(layers):
            ptrs = []
            for name in ("ln1", "wqkv", "bqkv", "wo", "ln2", "wgu", "wd"):
                t = w.get(name)
                if t is None:
                    if name != "bqkv":
                        raise ValueError(f"layer {i}: {name} missing")
                    ptrs.append(None)
                    continue
                if (t.dtype != torch.bfloat16 or not t.is_contiguous() or t.device != self.device):
                    raise ValueError(f"layer {i}: {name} must be contiguous bf16 on the device")
                keep.append(t)
                ptrs.append(t.data_ptr())
            W[i] = _abi.LayerWeights(*ptrs)
        nbytes = self.forward_workspace_bytes(R, params)
        ws = workspace if workspace is not None else self._fw_workspace(nbytes)
        fp = params.abi()
        with torch.cuda.device(self.device):
            _check(_lib().ss_question_forward(
                self.handle, W, C.byref(fp), C.c_void_p(h_in.data_ptr()), R,
                C.c_void_p(q_out.data_ptr()), C.c_void_p(h_out.data_ptr()),
                C.c_void_p(status.data_ptr() if status is not None else None),
                C.c_void_p(ws.data_ptr()), ws.numel(), C.c_void_p(_stream_ptr(self.device))))
        self._fw_keep = keep
        return q_out, h_out

    def _fw_workspace(self, nbytes: int) -> torch.Tensor:
        ws = getattr(self, "_fws", None)
        if ws is None or ws.numel() < nbytes:
            ws = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
            self._fws = ws
        return ws

    def compress(self, window_frames: int, n_centroids: int = 64, iters: int = 5,
                 first_frame: int = 0, n_frames: int | None = None) -> None:
        if n_frames is None:
            n_frames = (self.n_frames - first_frame) // window_frames * window_frames
        cp = _abi.CompressParams(window_frames, n_centroids, iters, first_frame, n_frames)
        with torch.cuda.device(self.device):
            _check(_lib().ss_index_compress(self.handle, C.byref(cp),
                                            C.c_void_p(_stream_ptr(self.device))))

    def workspace_bytes(self, n_rows: int, p: RetrieveParams) -> int:
        return workspace_bytes([self], [n_rows], p)

    def _workspace(self, nbytes: int) -> torch.Tensor:
        if self._ws is None or self._ws.numel() < nbytes:
            self._ws = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        return self._ws

    def retrieve(self, q: torch.Tensor, k: int, budget: int, *, pool_mult: int = 4,
                 n_prev: int = 1, n_recent: int = 0, q_agg: int = Q_LAST,
                 head_agg: int = H_PER_QHEAD, use_clusters: int = 0,
                 out: Result | None = None, workspace: torch.Tensor | None = None,
                 trace: tuple | None = None) -> Result:
        """One question against this index (Sec. 4.2, Eq. 10-12). q: bf16
        [P][R][Hq][128] on the index's device. Asynchronous on the current stream."""
        p = RetrieveParams(k, budget, pool_mult, n_prev, n_recent, q_agg, head_agg,
                           use_clusters)
        return retrieve_batched([self], [q], p, outs=[out] if out else None,
                                workspace=workspace, trace=trace)[0]

    def retrieve_static(self, q: torch.Tensor, p: RetrieveParams, out: Result) -> Result:
        """The retrieval of `retrieve` through ss_retrieve_static: the library allocates
        nothing and uses its fixed 64 MiB per-device scratch, for callers that cannot
        allocate device memory at question time. `out` is preallocated by the caller;
        calls on one device must not overlap (they share the scratch). Asynchronous on
        the current stream."""
        if q.dtype != torch.bfloat16 or q.dim() != 4 or not q.is_contiguous():
            raise ValueError("q must be contiguous bf16 [P][R][Hq][128]")
        if q.device != self.device:
            raise ValueError("q must be on the index's device")
        if q.shape[0] != self.n_layers or q.shape[2] != self.n_q_heads or q.shape[3] != 128:
            raise ValueError("q shape does not match the index")
        with torch.cuda.device(self.device):
            _check(_lib().ss_retrieve_static(self.handle, C.c_void_p(q.data_ptr()),
                                             q.shape[1], C.byref(p.to_c()),
                                             C.byref(out.to_c()),
                                             C.c_void_p(_stream_ptr(self.device))))
        out._keep = (q,)
        return out

    def retrieve_shard(self, q: torch.Tensor, p: RetrieveParams, unit_begin: int,
                       workspace: torch.Tensor | None = None) -> dict:
        """This index as one shard (stream units from unit_begin) of a retrieval split by
        token range: ss_retrieve_shard. Returns device tensors: topk_tok (stream ids),
        topk_s, list_stats, unit_stats, status; the descriptors are descriptors()."""
        if q.dtype != torch.bfloat16 or q.dim() != 4 or not q.is_contiguous() or q.device != self.device:
            raise ValueError("q must be contiguous bf16 [P][R][Hq][128] on the index's device")
        n_lists = self.n_layers * self.n_q_heads
        uh = max(0, self.n_units - p.n_recent)
        dev = self.device
        out = {"topk_tok": torch.empty(n_lists, p.k, dtype=torch.int32, device=dev),
               "topk_s": torch.empty(n_lists, p.k, dtype=torch.float32, device=dev),
               "list_stats": torch.empty(n_lists, 2, dtype=torch.float32, device=dev),
               "unit_stats": torch.empty(n_lists, max(uh, 1), 2, dtype=torch.float32, device=dev),
               "status": torch.zeros(1, dtype=torch.int32, device=dev)}
        nbytes = self.workspace_bytes(q.shape[1], p)
        ws = workspace if workspace is not None else self._workspace(nbytes)
        sr = _abi.ShardResult(*[out[k].data_ptr() for k in ("topk_tok", "topk_s", "list_stats",
                                                             "unit_stats", "status")])
        with torch.cuda.device(dev):
            _check(_lib().ss_retrieve_shard(self.handle, C.c_void_p(q.data_ptr()), q.shape[1],
                                            C.byref(p.to_c()), int(unit_begin), C.byref(sr),
                                            C.c_void_p(ws.data_ptr()), ws.numel(),
                                            C.c_void_p(_stream_ptr(dev))))
        out["unit_stats"] = out["unit_stats"][:, :uh]
        out["unit_begin"], out["n_units"] = int(unit_begin), uh
        out["_keep"] = (q, ws)
        return out

    def retrieve_host(self, q_host: torch.Tensor, p: RetrieveParams,
                      workspace: torch.Tensor | None = None) -> dict:
        """ss_retrieve_host: q in (pinned) host memory, selection copied back to host."""
        if q_host.device.type != "cpu" or q_host.dtype != torch.bfloat16:
            raise ValueError("q_host must be a bf16 CPU tensor")
        if not q_host.is_contiguous():
            q_host = q_host.contiguous()
        R = q_host.shape[1]
        # per (rows, params): the C parameter block, the workspace size and the host result
        # buffers (the call unpacks into them and they are copied out before returning)
        key = (R, p.k, p.budget, p.pool_mult, p.n_prev, p.n_recent, p.q_agg, p.head_agg,
               p.use_clusters)
        cached = self._host_calls.get(key)
        if cached is None:
            nexp = p.budget * (1 + p.n_prev)
            bufs = (torch.empty(p.budget, dtype=torch.int32),
                    torch.empty(nexp, dtype=torch.int32),
                    torch.empty(nexp * self.frames_per_unit, dtype=torch.int32),
                    torch.empty(4, dtype=torch.int32))
            hr = _abi.HostResult(*[b.data_ptr() for b in bufs])
            cached = (p.to_c(), self.workspace_bytes(R, p), bufs, hr)
            self._host_calls[key] = cached
        pc, nbytes, (sel, exp, frames, counts), hr = cached
        ws = workspace if workspace is not None else self._workspace(nbytes)
        _check(_lib().ss_retrieve_host(self.handle, q_host.data_ptr(), R, C.byref(pc),
                                       C.byref(hr), ws.data_ptr(), ws.numel(),
                                       torch.cuda.current_stream(self.device).cuda_stream))
        c = counts.tolist()
        return {"sel": sel.tolist()[:c[1]], "expanded": exp.tolist()[:c[2]],
                "frames": frames.tolist()[:c[3]], "counts": c}


def workspace_bytes(indexes: list[Index], n_rows: list[int], p: RetrieveParams) -> int:
    n = len(indexes)
    hs = (C.c_void_p * n)(*[ix.handle.value for ix in indexes])
    rs = (C.c_int32 * n)(*n_rows)
    out = C.c_size_t()
    _check(_lib().ss_retrieve_workspace_size(hs, n, rs, C.byref(p.to_c()), C.byref(out)))
    return out.value


def retrieve_batched(indexes: list[Index], qs: list[torch.Tensor], p: RetrieveParams,
                     outs: list[Result] | None = None, workspace: torch.Tensor | None = None,
                     trace: tuple | None = None) -> list[Result]:
    """n questions against n indexes on one device in one launch per stage."""
    n = len(indexes)
    if n != len(qs) or n == 0:
        raise ValueError("need one query per index")
    dev = indexes[0].device
    for ix, q in zip(indexes, qs):
        if q.dtype != torch.bfloat16 or q.dim() != 4 or not q.is_contiguous():
            raise ValueError("q must be contiguous bf16 [P][R][Hq][128]")
        if q.device != dev or ix.device != dev:
            raise ValueError("indexes and queries must share one device")
        if q.shape[0] != ix.n_layers or q.shape[2] != ix.n_q_heads or q.shape[3] != 128:
            raise ValueError("q shape does not match the index")
    rows = [q.shape[1] for q in qs]
    nbytes = workspace_bytes(indexes, rows, p)
    if workspace is None:
        workspace = indexes[0]._workspace(nbytes)
    if workspace.numel() * workspace.element_size() < nbytes:
        raise ValueError(f"workspace smaller than {nbytes} bytes")
    outs = outs or [Result(ix, p) for ix in indexes]
    hs = (C.c_void_p * n)(*[ix.handle.value for ix in indexes])
    qa = (C.c_void_p * n)(*[q.data_ptr() for q in qs])
    rs = (C.c_int32 * n)(*rows)
    res = (_abi.Result * n)(*[o.to_c() for o in outs])
    tr = None
    if trace is not None:
        tr = C.byref(_abi.Trace(trace[0].cuda_event if trace[0] is not None else None,
                                trace[1].cuda_event if trace[1] is not None else None))
    with torch.cuda.device(dev):
        _check(_lib().ss_retrieve_batched(hs, qa, rs, n, C.byref(p.to_c()), res,
                                          C.c_void_p(workspace.data_ptr()),
                                          workspace.numel() * workspace.element_size(),
                                          C.c_void_p(_stream_ptr(dev)), tr))
    for o in outs:
        o._keep = (workspace, qs)
    return outs


def merge_shards(shards: list[dict], n_lists: int, tokens_per_unit: int, p: RetrieveParams,
                 frames_per_unit: int = 1) -> dict:
    """ss_merge_shards on the host: the shards' payloads (numpy arrays or CPU tensors with
    keys unit_begin, n_units, topk_tok int32 [n_lists][k], topk_s fp32 [n_lists][k],
    list_stats fp32 [n_lists][2], unit_stats fp32 [n_lists][n_units][2], desc fp32
    [n_units][D]), in stream order. Returns numpy arrays of the merged retrieval."""
    import numpy as np

    def arr(x, dt):
        if isinstance(x, torch.Tensor):
            x = x.detach().cpu().numpy()
        return np.ascontiguousarray(x, dtype=dt)

    keep = []
    cs = (_abi.Shard * len(shards))()
    D = None
    for j, sh in enumerate(shards):
        a = [arr(sh["topk_tok"], np.int32), arr(sh["topk_s"], np.float32),
             arr(sh["list_stats"], np.float32), arr(sh["unit_stats"], np.float32),
             arr(sh["desc"], np.float32)]
        keep.append(a)
        D = a[4].shape[1] if a[4].ndim == 2 and a[4].shape[0] else (D or 1)
        cs[j] = _abi.Shard(int(sh["unit_begin"]), int(sh["n_units"]),
                           *[x.ctypes.data for x in a])
    U = sum(int(sh["n_units"]) for sh in shards)
    nexp = p.budget * (1 + p.n_prev)
    out = {"topk_tok": np.empty((n_lists, p.k), np.int32), "topk_w": np.empty((n_lists, p.k), np.float32),
           "list_stats": np.empty((n_lists, 2), np.float32), "votes": np.empty(U, np.int32),
           "mass": np.empty(U, np.float32), "pool": np.empty(max(1, min(p.pool_mult * p.budget, U)), np.int32),
           "sel": np.empty(p.budget, np.int32), "expanded": np.empty(nexp, np.int32),
           "frames": np.empty(nexp * frames_per_unit, np.int32), "counts": np.zeros(4, np.int32)}
    mr = _abi.MergeResult(*[out[k].ctypes.data for k in ("topk_tok", "topk_w", "list_stats",
                                                         "votes", "mass", "pool", "sel",
                                                         "expanded", "frames", "counts")])
    _check(_lib().ss_merge_shards(cs, len(shards), n_lists, tokens_per_unit, frames_per_unit,
                                  int(D or 1), C.byref(p.to_c()), C.byref(mr)))
    c = out["counts"]
    out["pool"], out["sel"] = out["pool"][:c[0]], out["sel"][:c[1]]
    out["expanded"], out["frames"] = out["expanded"][:c[2]], out["frames"][:c[3]]
    return out
