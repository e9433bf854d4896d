"""Failure paths of the C ABI, made on the host or by a wait limit, with no GPU fault:

* an allocator that returns NULL on its n-th call makes ss_index_create and
  ss_index_compress fail with SS_ERR_ALLOC and give back every block they took;
* a wait limit of 0 polls makes the key-scoring kernel's waits for its key copies give
  up: the retrieval reports SS_ERR_TIMEOUT (through ss_status_sync and
  ss_retrieve_host), its later kernels skip their work, and the next retrieval with the
  default limit is correct again (the context stays usable).
"""
import ctypes as C

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


class CountingAllocator:
    """ss_allocator backed by torch tensors that fails (returns NULL) on call `fail_at`."""

    def __init__(self, fail_at: int | None):
        from paper_2609_02780_gb300 import _abi
        self.fail_at = fail_at
        self.calls = 0
        self.live: dict[int, torch.Tensor] = {}
        self.freed = 0
        self._a = _abi.ALLOC_FN(self._alloc)
        self._f = _abi.FREE_FN(self._free)
        self.c = _abi.Allocator(self._a, self._f, None)

    def _alloc(self, nbytes, stream, ctx):
        self.calls += 1
        if self.fail_at is not None and self.calls == self.fail_at:
            return None
        t = torch.empty(int(nbytes), dtype=torch.uint8, device="cuda")
        self.live[t.data_ptr()] = t
        return t.data_ptr()

    def _free(self, ptr, stream, ctx):
        assert ptr in self.live, "free of a block this allocator did not hand out"
        del self.live[ptr]
        self.freed += 1


def _cfg():
    from paper_2609_02780_gb300 import _abi
    return _abi.IndexConfig(2, 8, 2, 128, 16, 1, 40)


def _stream():
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def test_create_allocation_failure_releases_everything():
    ss = _ss()
    lib = ss._abi.load()
    cfg = _cfg()
    probe = CountingAllocator(None)
    h = C.c_void_p()
    assert lib.ss_index_create(C.byref(cfg), C.byref(probe.c), _stream(), C.byref(h)) == 0
    n_create = probe.calls
    assert n_create >= 2
    assert lib.ss_index_destroy(h) == 0
    assert not probe.live
    for n in range(1, n_create + 1):
        a = CountingAllocator(n)
        h = C.c_void_p()
        st = lib.ss_index_create(C.byref(cfg), C.byref(a.c), _stream(), C.byref(h))
        assert st == 5, (n, st)                        # SS_ERR_ALLOC
        assert not h.value
        assert not a.live, f"allocation {n} failed: {len(a.live)} blocks leaked"
        assert b"allocation" in lib.ss_last_error()


def test_compress_allocation_failure_leaves_a_usable_index():
    ss = _ss()
    lib = ss._abi.load()
    cfg = _cfg()
    g = torch.Generator().manual_seed(5)
    keys = torch.randn(2, 2, 40 * 16, 128, generator=g).to(torch.bfloat16).cuda()
    probe = CountingAllocator(None)
    h = C.c_void_p()
    assert lib.ss_index_create(C.byref(cfg), C.byref(probe.c), _stream(), C.byref(h)) == 0
    assert lib.ss_index_append(h, C.c_void_p(keys.data_ptr()), 40, 0, _stream()) == 0
    cp = ss._abi.CompressParams(4, 8, 2, 0, 20)
    n_create = probe.calls
    assert lib.ss_index_compress(h, C.byref(cp), _stream()) == 0
    n_compress = probe.calls - n_create
    assert n_compress >= 2
    assert lib.ss_index_destroy(h) == 0
    assert not probe.live
    for n in range(1, n_compress + 1):
        a = CountingAllocator(n_create + n)
        h = C.c_void_p()
        assert lib.ss_index_create(C.byref(cfg), C.byref(a.c), _stream(), C.byref(h)) == 0
        assert lib.ss_index_append(h, C.c_void_p(keys.data_ptr()), 40, 0, _stream()) == 0
        before = dict(a.live)
        assert lib.ss_index_compress(h, C.byref(cp), _stream()) == 5, n   # SS_ERR_ALLOC
        assert set(a.live) == set(before), "a failed compression kept cluster blocks"
        v = ss._abi.IndexView()
        assert lib.ss_index_get_view(h, C.byref(v)) == 0
        assert v.n_windows == 0 and v.window_frames == 0 and not v.centroids
        # with memory available again the same compression succeeds
        a.fail_at = None
        assert lib.ss_index_compress(h, C.byref(cp), _stream()) == 0
        assert lib.ss_index_get_view(h, C.byref(v)) == 0
        assert v.n_windows == 5
        torch.cuda.synchronize()
        assert lib.ss_index_destroy(h) == 0
        assert not a.live


def _small_index():
    ss = _ss()
    g = torch.Generator().manual_seed(9)
    P, Hq, Hkv, F, Tf = 2, 8, 2, 60, 50
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g).to(torch.bfloat16)
    q = torch.randn(P, 3, Hq, 128, generator=g).to(torch.bfloat16)
    idx = ss.Index(P, Hq, Hkv, Tf, F, device="cuda")
    idx.append(keys.cuda())
    return idx, q


def test_score_wait_timeout_is_reported_and_the_context_recovers():
    ss = _ss()
    lib = ss._abi.load()
    idx, q = _small_index()
    p = ss.RetrieveParams(k=64, budget=4)
    good = idx.retrieve(q.cuda(), k=p.k, budget=p.budget)
    good_host = good.host()
    assert lib.ss_set_wait_limit(-2) == 1               # rejected: INVALID_ARG
    try:
        assert lib.ss_set_wait_limit(0) == 0
        res = idx.retrieve(q.cuda(), k=p.k, budget=p.budget)
        with pytest.raises(ss.ShallowStreamError, match="TIMEOUT"):
            res.check()
        # the later kernels skipped their work: no pool, no selection
        assert res.counts.cpu().tolist() == [0, 0, 0, 0]
        with pytest.raises(ss.ShallowStreamError, match="TIMEOUT"):
            idx.retrieve_host(q, p)
    finally:
        assert lib.ss_set_wait_limit(-1) == 0
    again = idx.retrieve(q.cuda(), k=p.k, budget=p.budget)
    assert again.host() == good_host
    assert torch.equal(again.topk_tok, good.topk_tok)
    assert idx.retrieve_host(q, p)["frames"] == good_host["frames"]
