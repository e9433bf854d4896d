"""Checkpoint of an index (ss_index_save / ss_index_load): a loaded index retrieves, keeps
compressing and clustering, and runs the question's forward exactly as the saved one."""
import os

import pytest
import torch

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _same(a, b, n_units):
    """Equal lists, statistics and selection; per-unit arrays over the stored units (the
    entries past them are not written by a retrieval)."""
    for f in ("topk_tok", "topk_w", "list_stats", "counts"):
        assert torch.equal(getattr(a, f), getattr(b, f)), f
    for f in ("unit_votes", "unit_mass"):
        assert torch.equal(getattr(a, f)[:n_units], getattr(b, f)[:n_units]), f
    assert a.host() == b.host()


def _data(seed, P=2, Hkv=4, F=48, Tf=64, R=8):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g).to(torch.bfloat16).cuda()
    vals = torch.randn(P, Hkv, F * Tf, 128, generator=g).to(torch.bfloat16).cuda()
    q = torch.randn(P, R, Hkv * 7, 128, generator=g).to(torch.bfloat16).cuda()
    return keys, vals, q


def test_plain_index_with_values_round_trip(tmp_path):
    ss = _ss()
    keys, vals, q = _data(1)
    idx = ss.Index(2, 28, 4, 64, 64, frames_per_unit=2, device="cuda")
    idx.append(keys)
    idx.append_values(vals)
    path = os.path.join(tmp_path, "a.ssidx")
    idx.save(path)
    ld = ss.Index.load(path)
    assert (ld.n_layers, ld.n_q_heads, ld.n_kv_heads, ld.tokens_per_frame,
            ld.frames_per_unit, ld.max_frames) == (2, 28, 4, 64, 2, 64)
    assert ld.n_frames == 48 and ld.n_units == 24
    assert torch.equal(ld.keys(), idx.keys()) and torch.equal(ld.values(), idx.values())
    assert torch.equal(ld.descriptors(), idx.descriptors())
    _same(idx.retrieve(q, k=200, budget=5, n_recent=2), ld.retrieve(q, k=200, budget=5, n_recent=2),
          22)
    # both keep appending the same frames and agree
    more, mv, _ = _data(2, F=16)
    for ix in (idx, ld):
        ix.append(more)
        ix.append_values(mv)
    _same(idx.retrieve(q, k=300, budget=6), ld.retrieve(q, k=300, budget=6), 32)


def test_compressed_windows_round_trip(tmp_path):
    ss = _ss()
    keys, _, q = _data(3)
    idx = ss.Index(2, 28, 4, 64, 80, device="cuda")
    idx.append(keys)
    idx.compress(8, n_centroids=16, iters=3, first_frame=8, n_frames=16)
    path = os.path.join(tmp_path, "b.ssidx")
    idx.save(path)
    ld = ss.Index.load(path)
    a, b = idx.clusters(), ld.clusters()
    for k in ("centroids", "member_counts", "member_sizes", "window_first_unit"):
        assert torch.equal(a[k], b[k]), k
    _same(idx.retrieve(q, k=64, budget=4, use_clusters=1), ld.retrieve(q, k=64, budget=4, use_clusters=1),
          48)
    # compression continues after the loaded windows
    for ix in (idx, ld):
        ix.compress(8, n_centroids=16, iters=3, first_frame=24, n_frames=16)
    _same(idx.retrieve(q, k=64, budget=4, use_clusters=1), ld.retrieve(q, k=64, budget=4, use_clusters=1),
          48)


def test_unit_clusters_round_trip(tmp_path):
    ss = _ss()
    keys, _, q = _data(4)
    idx = ss.Index(2, 28, 4, 64, 48, device="cuda")
    idx.append(keys)
    idx.cluster_units(20, 0.1, max_clusters=32)
    path = os.path.join(tmp_path, "c.ssidx")
    idx.save(path)
    ld = ss.Index.load(path)
    a, b = idx.unit_clusters(), ld.unit_clusters()
    for k in ("unit_cluster", "centroids", "sizes", "keys"):
        assert torch.equal(a[k], b[k]), k
    _same(idx.retrieve(q, k=100, budget=4), ld.retrieve(q, k=100, budget=4), 48)
    ra, rb = idx.select_clusters(q, k_l=4), ld.select_clusters(q, k_l=4)
    assert torch.equal(ra["ids"], rb["ids"]) and torch.equal(ra["scores"], rb["scores"])
    for ix in (idx, ld):
        ix.cluster_units(10, 0.1, max_clusters=32)
    a, b = idx.unit_clusters(), ld.unit_clusters()
    assert torch.equal(a["centroids"], b["centroids"]) and torch.equal(a["keys"], b["keys"])


def test_bad_files_are_rejected(tmp_path):
    ss = _ss()
    p = os.path.join(tmp_path, "x.ssidx")
    with open(p, "wb") as f:
        f.write(b"not an index")
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        ss.Index.load(p)
    keys, _, _ = _data(5, F=8)
    idx = ss.Index(2, 28, 4, 64, 8, device="cuda")
    idx.append(keys)
    good = os.path.join(tmp_path, "g.ssidx")
    idx.save(good)
    data = open(good, "rb").read()
    with open(p, "wb") as f:
        f.write(data[: len(data) // 2])
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        ss.Index.load(p)
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        ss.Index.load(os.path.join(tmp_path, "missing.ssidx"))
