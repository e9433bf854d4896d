"""Seeded synthetic shallow-index workloads.

Draws the bf16 keys that the shallow layers [0, P) of a streaming MLLM would archive
for a video stream (Sec. 4.1, Eq. 1-2) and the post-RoPE query rows of a question at
those layers (Sec. 4.2, Eq. 10), shaped like the 1 fps streams of Sec. 5.1 and the
settings of Table 4. The paper's benchmarks and model weights are not used; these
tensors stand in for them.

This module only draws random numbers and lays them out. It holds none of the
retrieval arithmetic, so both the CUDA path's tests and the CPU oracle's tests can
consume its bytes.

Layouts (all contiguous, bf16):
  keys    [P][Hkv][F * T_f][d]   token id p = frame * T_f + slot
  values  [P][Hkv][F * T_f][d]   (the question's forward only)
  queries [P][R][Hq][d]
  question rows [R][Hq d] and decoder-layer weights (the question's forward only)
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int                 # P, shallow layers
    n_frames: int                 # F
    tokens_per_frame: int         # T_f
    n_rows: int                   # R, question rows
    k: int                        # top-k per list
    budget: int                   # K, units selected before expansion
    n_planted: int
    keys: str                     # "offset" | "drift_outlier" | "scenes" | "iid"
    seed: int = 0
    n_q_heads: int = 28
    n_kv_heads: int = 4
    head_dim: int = 128
    frames_per_unit: int = 1
    pool_mult: int = 4
    n_prev: int = 1
    n_recent: int = 0
    q_agg: int = 0                # 0 = last row, 1 = mean of rows (mean logit)
    head_agg: int = 0             # 0 = per query head, 1 = mean over heads
    # k-means compression (0 windows = none)
    window_frames: int = 0
    n_centroids: int = 64
    kmeans_iters: int = 5
    n_streams: int = 1            # >1: independent streams, seeds seed..seed+n-1
    extra: dict = field(default_factory=dict, compare=False)

    @property
    def tokens_per_unit(self) -> int:
        return self.tokens_per_frame * self.frames_per_unit

    @property
    def n_units(self) -> int:
        return self.n_frames // self.frames_per_unit

    @property
    def n_tokens(self) -> int:
        return self.n_frames * self.tokens_per_frame

    @property
    def n_slabs(self) -> int:
        return self.n_layers * self.n_kv_heads

    @property
    def n_hist_units(self) -> int:
        return max(0, self.n_units - self.n_recent)

    @property
    def keys_per_query(self) -> int:
        """Stored (layer, kv-head, token) key rows scored by one query."""
        return self.n_slabs * self.n_hist_units * self.tokens_per_unit

    @property
    def key_bytes(self) -> int:
        return self.n_slabs * self.n_tokens * self.head_dim * 2

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# Named workloads. Shapes follow the streams described for evaluation (1 fps, Sec. 5.1)
# and the evidence-selection settings of Table 4 (pool = 4K, one preceding unit).
PRESETS = {
    "tiny": Workload("tiny", n_layers=2, n_frames=64, tokens_per_frame=64, n_rows=16,
                     k=256, budget=8, n_planted=4, keys="offset", seed=0),
    "hour1": Workload("hour1", n_layers=4, n_frames=3600, tokens_per_frame=196,
                      n_rows=32, k=1024, budget=64, n_planted=16,
                      keys="drift_outlier", seed=0),
    "hour1_kmeans": Workload("hour1_kmeans", n_layers=4, n_frames=3600,
                             tokens_per_frame=196, n_rows=32, k=512, budget=64,
                             n_planted=16, keys="drift_outlier", seed=0,
                             window_frames=20),
    "hour3": Workload("hour3", n_layers=6, n_frames=5400, tokens_per_frame=256,
                      n_rows=64, k=2048, budget=96, n_planted=24, keys="scenes", seed=0),
    "batched16": Workload("batched16", n_layers=4, n_frames=1800, tokens_per_frame=196,
                          n_rows=32, k=1024, budget=48, n_planted=16,
                          keys="drift_outlier", seed=0, n_streams=16),
    # the 1-hour stream with lists ranked by the mean of all 32 question rows' softmax
    # weights (every row attends on its own)
    "hour1_msm": Workload("hour1_msm", n_layers=4, n_frames=3600, tokens_per_frame=196,
                          n_rows=32, k=1024, budget=64, n_planted=16,
                          keys="drift_outlier", seed=0, q_agg=2),
    # the 1-hour stream with the question's forward through the shallow layers (Eq. 10):
    # synthetic decoder layers of hidden size 28 * 128 and MLP width 18944 produce the
    # query rows the retrieval scores
    "hour1_fwd": Workload("hour1_fwd", n_layers=4, n_frames=3600, tokens_per_frame=196,
                          n_rows=32, k=1024, budget=64, n_planted=16,
                          keys="drift_outlier", seed=0, extra={"intermediate": 18944}),
    # Table 4 evidence-selection settings (Qwen3-VL column: 2-frame units, P = 5,
    # 64 candidates per layer averaged over heads, pool 32, K = 8, 6 recent units).
    "paper_qwen": Workload("paper_qwen", n_layers=5, n_frames=256, tokens_per_frame=64,
                           n_rows=8, k=64, budget=8, n_planted=4, keys="offset",
                           seed=0, frames_per_unit=2, n_recent=6, head_agg=1),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def make_queries(w: Workload, device="cpu", seed: int | None = None) -> torch.Tensor:
    """Question query rows, bf16 [P][R][Hq][d], ~N(0, 1)."""
    g = _gen(w.seed if seed is None else seed, device)
    q = torch.randn(w.n_layers, w.n_rows, w.n_q_heads, w.head_dim, generator=g,
                    device=device, dtype=torch.float32)
    return q.to(torch.bfloat16)


def planted_frames(w: Workload, seed: int | None = None) -> list[int]:
    """Frames whose keys are shifted toward the question (sorted)."""
    s = (w.seed if seed is None else seed)
    rng = np.random.default_rng(10_007 + s)
    hist_frames = w.n_hist_units * w.frames_per_unit
    if hist_frames <= 0 or w.n_planted <= 0:
        return []
    if w.keys == "scenes":
        scene_len = int(w.extra.get("scene_frames", 120))
        n_scenes = max(1, hist_frames // scene_len)
        per_scene = 3
        n_pick = max(1, min(n_scenes, w.n_planted // per_scene))
        scenes = rng.choice(n_scenes, size=n_pick, replace=False)
        out = []
        for sc in scenes:
            lo = sc * scene_len
            hi = min(hist_frames, lo + scene_len)
            out += list(rng.choice(np.arange(lo, hi), size=min(per_scene, hi - lo),
                                   replace=False))
        return sorted(int(f) for f in out)
    n = min(w.n_planted, hist_frames)
    return sorted(int(f) for f in rng.permutation(hist_frames)[:n])


def _planted_shift(w: Workload, q: torch.Tensor) -> torch.Tensor:
    """0.5 * mean over each GQA group's query heads of the last question row:
    fp32 [P][Hkv][d]."""
    G = w.n_q_heads // w.n_kv_heads
    last = q[:, -1].float().reshape(w.n_layers, w.n_kv_heads, G, w.head_dim)
    return 0.5 * last.mean(dim=2)


def make_keys(w: Workload, q: torch.Tensor, device="cpu",
              seed: int | None = None) -> torch.Tensor:
    """Shallow keys, bf16 [P][Hkv][F*T_f][d].

    Draw order: per layer, per kv head, then frames. Value recipes:
      offset         N(0,1) + a per-frame offset vector ~ N(0, 0.3^2)
      drift_outlier  N(0,1) with 2 seeded channels x8, + an AR(1) per-frame mean
                     (rho 0.98, innovation std 0.06, stationary std 0.3)
      scenes         N(0,1) + a scene mean ~ N(0, 0.5^2), new scene every 120 frames
      iid            N(0,1)
    Planted frames add 0.5 * (mean of the group's last-row query heads) to every token.
    """
    s = w.seed if seed is None else seed
    g = _gen(1_000_003 + s, device)
    P, Hkv, F, Tf, d = w.n_layers, w.n_kv_heads, w.n_frames, w.tokens_per_frame, w.head_dim
    out = torch.empty(P, Hkv, F * Tf, d, dtype=torch.bfloat16, device=device)
    shift = _planted_shift(w, q.to(device))
    planted = planted_frames(w, s)
    frame_of_tok = torch.arange(F, device=device).repeat_interleave(Tf)
    for i in range(P):
        for j in range(Hkv):
            z = torch.randn(F * Tf, d, generator=g, device=device, dtype=torch.float32)
            if w.keys == "offset":
                off = 0.3 * torch.randn(F, d, generator=g, device=device)
                z += off[frame_of_tok]
            elif w.keys == "drift_outlier":
                ch = torch.randperm(d, generator=g, device=device)[:2]
                z[:, ch] *= 8.0
                mu0 = 0.3 * torch.randn(d, generator=g, device=device)
                innov = 0.06 * torch.randn(F, d, generator=g, device=device)
                mu = np.empty((F, d), dtype=np.float64)
                prev = mu0.double().cpu().numpy()
                inn = innov.double().cpu().numpy()
                for f in range(F):
                    prev = (0.98 * prev + inn[f]) if f > 0 else prev
                    mu[f] = prev
                z += torch.from_numpy(mu).float().to(device)[frame_of_tok]
            elif w.keys == "scenes":
                scene_len = int(w.extra.get("scene_frames", 120))
                n_sc = (F + scene_len - 1) // scene_len
                sm = 0.5 * torch.randn(n_sc, d, generator=g, device=device)
                z += sm[frame_of_tok // scene_len]
            elif w.keys != "iid":
                raise ValueError(f"unknown key recipe {w.keys!r}")
            for f in planted:
                z[f * Tf:(f + 1) * Tf] += shift[i, j]
            out[i, j] = z.to(torch.bfloat16)
    return out


def make_values(w: Workload, device="cpu", seed: int | None = None) -> torch.Tensor:
    """Shallow values, bf16 [P][Hkv][F*T_f][d] ~ N(0, 1), drawn per layer, per kv head."""
    s = w.seed if seed is None else seed
    g = _gen(2_000_003 + s, device)
    P, Hkv, N, d = w.n_layers, w.n_kv_heads, w.n_frames * w.tokens_per_frame, w.head_dim
    out = torch.empty(P, Hkv, N, d, dtype=torch.bfloat16, device=device)
    for i in range(P):
        for j in range(Hkv):
            out[i, j] = torch.randn(N, d, generator=g, device=device).to(torch.bfloat16)
    return out


def make_forward_weights(w: Workload, intermediate: int, device="cpu", seed: int | None = None,
                         bias: bool = True) -> list[dict]:
    """Synthetic weights of the P shallow decoder layers (one dict per layer, bf16):
    RMSNorm weights 1 + N(0, 0.1^2); projections N(0, 1 / fan_in); q/k/v bias N(0, 0.1^2).
    Layouts as ss_layer_weights: wqkv [(Hq + 2 Hkv) d][D], wo [D][Hq d], wgu [2 I][D]
    (gate rows, then up rows), wd [D][I]."""
    s = w.seed if seed is None else seed
    g = _gen(3_000_017 + s, device)
    D = w.n_q_heads * w.head_dim
    nqkv = (w.n_q_heads + 2 * w.n_kv_heads) * w.head_dim
    I = intermediate

    def rnd(*shape, std=1.0, mean=0.0):
        x = torch.randn(*shape, generator=g, device=device) * std + mean
        return x.to(torch.bfloat16).contiguous()

    layers = []
    for _ in range(w.n_layers):
        layers.append({
            "ln1": rnd(D, std=0.1, mean=1.0),
            "wqkv": rnd(nqkv, D, std=D ** -0.5),
            "bqkv": rnd(nqkv, std=0.1) if bias else None,
            "wo": rnd(D, D, std=D ** -0.5),
            "ln2": rnd(D, std=0.1, mean=1.0),
            "wgu": rnd(2 * I, D, std=D ** -0.5),
            "wd": rnd(D, I, std=I ** -0.5),
        })
    return layers


def make_question_rows(w: Workload, device="cpu", seed: int | None = None) -> torch.Tensor:
    """The question's embedded rows entering the first shallow layer, bf16 [R][Hq d] ~ N(0, 1)."""
    s = w.seed if seed is None else seed
    g = _gen(4_000_037 + s, device)
    D = w.n_q_heads * w.head_dim
    return torch.randn(w.n_rows, D, generator=g, device=device).to(torch.bfloat16)


def make_workload(w: Workload, device="cpu", stream: int = 0) -> dict:
    """Keys, queries and planted frames of one stream (seed = w.seed + stream)."""
    s = w.seed + stream
    q = make_queries(w, device, seed=s)
    keys = make_keys(w, q, device, seed=s)
    return {"keys": keys, "q": q, "planted": planted_frames(w, s), "seed": s}


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw bf16 bit patterns of a tensor as a numpy uint16 array (host copy)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
