"""Parity of the k-means compression kernel (through the C ABI) with the CPU oracle.

Lloyd rounds are chained: the GPU's assignment after round t is checked against the
fp64 nearest centroid of the oracle's centroids C_{t-1}, themselves the fp64 means of
the GPU's assignment after round t - 1 (C_0 = the window's first n_c keys); the GPU's
stored centroids after round t against the fp64 means of its own round-t assignment.
A run with `iters = t` is the first t rounds of a longer run (the kernel is
deterministic), so one index per t gives every round.

Distance tolerance: both kernels (tcgen05 for n_c <= 64, mma.sync above) compare
||c||^2 - 2 x . c in fp32, with x . c on the tensor cores from c split into two bf16
parts (|c - c_hi - c_lo| <= 2^-18 |c| per element) and 256 products accumulated in fp32
(<= 256 * 2^-23 relative), and ||c||^2 as a 128-term fp32 sum. Each distance is then
off by at most about 3e-5 * (||x||^2 + ||c||^2); a difference of two by twice that.
TOL_REL = 1e-4 covers it. The member sums behind each mean are fp32 sums of exact
bf16 keys (tensor-core accumulation on the tcgen05 path), far inside the half-ulp bound
the stored bf16 centroids are checked with.
"""
import numpy as np
import pytest
import torch

from oracle import kmeans as KM
from oracle import retrieval as R

pytestmark = pytest.mark.gpu

TOL_REL = 1e-4


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _index(keys, Tf, fpu=1):
    import paper_2609_02780_gb300 as ss
    P, Hkv, N, _ = keys.shape
    idx = ss.Index(P, Hkv * 2, Hkv, Tf, N // Tf, frames_per_unit=fpu, device="cuda")
    idx.append(keys.cuda())
    return idx


def _gpu_round(keys, Tf, WF, n_c, iters, fpu=1):
    idx = _index(keys, Tf, fpu)
    idx.compress(WF, n_centroids=n_c, iters=iters)
    cl = idx.clusters()
    torch.cuda.synchronize()
    return {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in cl.items()}


def _check_assignment(X, C_prev, a_gpu):
    """GPU picks are nearest up to the rounding band; returns the ambiguous count."""
    D = ((X[:, None, :] - C_prev[None, :, :]) ** 2).sum(-1)
    best = D.min(1)
    tol = TOL_REL * ((X * X).sum(1) + (C_prev * C_prev).sum(1).max())
    got = D[np.arange(len(X)), a_gpu]
    assert (got <= best + tol).all(), "a key is not assigned to a (near-)nearest centroid"
    ref = D.argmin(1)
    srt = np.sort(D, axis=1)
    gap = srt[:, 1] - srt[:, 0] if D.shape[1] > 1 else np.full(len(X), np.inf)
    clear = gap > tol
    assert (a_gpu[clear] == ref[clear]).all(), "assignment differs where the gap is clear"
    return int((~clear).sum())


def _means(X, a, C_prev):
    C = C_prev.copy()
    for c in range(C.shape[0]):
        m = a == c
        if m.any():
            C[c] = X[m].mean(0)
    return C


def _chained(keys, Tf, WF, n_c, T, fpu=1):
    P, Hkv, N, _ = keys.shape
    kb = _bits(keys)
    Wt = WF * Tf
    n_w = N // Wt
    rounds = [_gpu_round(keys, Tf, WF, n_c, t, fpu) for t in range(1, T + 1)]
    ambiguous = total = 0
    for i in range(P):
        for g in range(Hkv):
            for w in range(n_w):
                X = R.bf16_to_f64(kb[i, g, w * Wt:(w + 1) * Wt])
                C = X[:n_c].copy()
                for t, r in enumerate(rounds, start=1):
                    a = r["assignment"][i, g, w * Wt:(w + 1) * Wt].numpy().astype(np.int64)
                    ambiguous += _check_assignment(X, C, a)
                    total += len(a)
                    C = _means(X, a, C)
                    cg = R.bf16_to_f64(_bits(r["centroids"][i, g, w]))
                    assert np.all(np.abs(cg - C) <= 2.0 ** -8 * np.abs(C) + 1e-6), \
                        f"round {t}: stored centroid is not the bf16 mean of its members"
                # member counts of the last round, per unit of the window
                a = rounds[-1]["assignment"][i, g, w * Wt:(w + 1) * Wt].numpy()
                Tu = Tf * fpu
                cnt = np.zeros((n_c, WF // fpu), dtype=np.int64)
                np.add.at(cnt, (a.astype(np.int64), np.arange(Wt) // Tu), 1)
                assert np.array_equal(rounds[-1]["member_counts"][i, g, w].numpy(), cnt)
                assert np.array_equal(rounds[-1]["member_sizes"][i, g, w].numpy(), cnt.sum(1))
    return rounds, ambiguous / total


def test_lloyd_rounds_chained_against_the_oracle():
    g = torch.Generator().manual_seed(20)
    keys = torch.randn(2, 2, 24 * 40, 128, generator=g)
    keys[..., 5] *= 8.0                                    # an outlier channel
    keys = keys.to(torch.bfloat16)
    rounds, amb = _chained(keys, Tf=40, WF=4, n_c=12, T=4)   # 6 windows of 160 keys
    assert amb < 0.05
    wf = rounds[-1]["window_first_unit"].tolist()
    assert wf == [0, 4, 8, 12, 16, 20]


def test_hour_like_window_and_two_frame_units():
    # the 1-hour configuration's window (20 frames x 196 tokens, 64 centroids, 5 rounds)
    g = torch.Generator().manual_seed(21)
    keys = (torch.randn(1, 2, 40 * 196, 128, generator=g) +
            0.3 * torch.randn(1, 2, 40, 1, 128, generator=g).repeat_interleave(196, 2)
            .reshape(1, 2, 40 * 196, 128)).to(torch.bfloat16)
    _, amb = _chained(keys, Tf=196, WF=20, n_c=64, T=5, fpu=2)
    assert amb < 0.05


def test_identity_when_every_key_is_a_centroid():
    g = torch.Generator().manual_seed(22)
    keys = torch.randn(1, 1, 4 * 8, 128, generator=g).to(torch.bfloat16)
    r = _gpu_round(keys, Tf=8, WF=2, n_c=16, iters=3)
    for w in range(2):
        assert r["assignment"][0, 0, w * 16:(w + 1) * 16].tolist() == list(range(16))
        assert torch.equal(r["centroids"][0, 0, w], keys[0, 0, w * 16:(w + 1) * 16])


def test_well_separated_blobs_are_recovered():
    g = torch.Generator().manual_seed(23)
    centers = 20.0 * torch.randn(4, 128, generator=g)
    lab = torch.cat([torch.arange(4), torch.randint(0, 4, (60,), generator=g)])
    keys = (centers[lab] + 0.1 * torch.randn(64, 128, generator=g)).to(torch.bfloat16)
    r = _gpu_round(keys.view(1, 1, 64, 128), Tf=16, WF=4, n_c=4, iters=3)
    assert torch.equal(r["assignment"][0, 0, :64].long(), lab)
    X = keys.double()
    for c in range(4):
        m = X[lab == c].mean(0)
        cg = r["centroids"][0, 0, 0, c].double()
        assert torch.all((cg - m).abs() <= 2.0 ** -8 * m.abs() + 1e-6)


def test_incremental_windows_and_determinism():
    import paper_2609_02780_gb300 as ss
    g = torch.Generator().manual_seed(24)
    keys = torch.randn(2, 2, 30 * 20, 128, generator=g).to(torch.bfloat16)
    one = _gpu_round(keys, Tf=20, WF=5, n_c=8, iters=3)
    idx = _index(keys, 20)
    idx.compress(5, n_centroids=8, iters=3, first_frame=0, n_frames=10)
    idx.compress(5, n_centroids=8, iters=3, first_frame=10, n_frames=20)
    two = idx.clusters()
    for k in ("centroids", "assignment", "member_counts", "member_sizes", "window_first_unit"):
        assert torch.equal(one[k], two[k].cpu()), k
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        idx.compress(5, n_centroids=8, iters=3, first_frame=20, n_frames=5)   # overlap
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        _index(keys, 20).compress(5, n_centroids=129, iters=1)


def test_oracle_compress_agrees_on_a_clear_case():
    # with well separated data the whole oracle run and the GPU run agree exactly
    g = torch.Generator().manual_seed(25)
    centers = 10.0 * torch.randn(8, 128, generator=g)
    lab = torch.cat([torch.arange(8), torch.randint(0, 8, (152,), generator=g)])
    keys = (centers[lab] + 0.5 * torch.randn(160, 128, generator=g)).to(torch.bfloat16)
    keys = keys.view(1, 1, 160, 128)
    r = _gpu_round(keys, Tf=40, WF=4, n_c=8, iters=5)
    ref = KM.compress(_bits(keys), tokens_per_frame=40, first_frame=0, n_frames=4,
                      window_frames=4, n_centroids=8, iters=5)
    assert np.array_equal(r["assignment"][0, 0, :160].numpy(), ref["assign"][0, 0, 0])
    cg = _bits(r["centroids"][0, 0, 0]).astype(np.int64)
    cr = ref["centroid_bits"][0, 0, 0].astype(np.int64)
    assert np.abs(cg - cr).max() <= 1          # bf16 of an fp32 vs an fp64 mean


def test_more_than_64_centroids_take_the_mma_sync_kernel():
    # n_c = 96 is past the tcgen05 kernel's limit: the other kernel, same contract
    g = torch.Generator().manual_seed(26)
    keys = (torch.randn(1, 2, 12 * 50, 128, generator=g) +
            0.5 * torch.randn(1, 2, 12, 1, 128, generator=g).repeat_interleave(50, 2)
            .reshape(1, 2, 600, 128)).to(torch.bfloat16)
    _, amb = _chained(keys, Tf=50, WF=4, n_c=96, T=3)     # 3 windows of 200 keys
    assert amb < 0.05


def test_window_of_one_partial_tile_and_many_full_tiles():
    # 100-token windows (one ragged 128-token tile) and 1,300-token windows (10 full
    # tiles and a ragged one), 40 centroids (padded to 48 operand rows)
    g = torch.Generator().manual_seed(27)
    keys = torch.randn(1, 1, 26 * 100, 128, generator=g).to(torch.bfloat16)
    _, amb = _chained(keys, Tf=100, WF=1, n_c=40, T=3)
    assert amb < 0.05
    _, amb = _chained(keys, Tf=100, WF=13, n_c=40, T=3)
    assert amb < 0.05
