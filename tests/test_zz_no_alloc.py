"""The allocation-free retrieval entry point (ss_retrieve_static) against ss_retrieve.

Named to be collected last, so that it runs both after the rest of the GPU suite and,
when selected alone, with the library's per-device set-up done by its own first call.
"""
import gc

import pytest
import torch

pytestmark = pytest.mark.gpu

# whole arrays; the pool, selection and frames are compared over their valid prefixes
INT_OUTPUTS = ("topk_tok", "unit_votes", "counts")
FLOAT_OUTPUTS = ("topk_w", "list_stats", "unit_mass")


def _case(seed, P=2, Hq=8, Hkv=2, F=96, Tf=40, R=4):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g).to(torch.bfloat16)
    q = torch.randn(P, R, Hq, 128, generator=g).to(torch.bfloat16)
    return keys, q


def _same(a, b, uh):
    for name in INT_OUTPUTS:
        x, y = getattr(a, name), getattr(b, name)
        if name == "unit_votes":
            x, y = x[:uh], y[:uh]
        assert torch.equal(x, y), name
    for name in FLOAT_OUTPUTS:
        x, y = getattr(a, name), getattr(b, name)
        if name == "unit_mass":
            x, y = x[:uh], y[:uh]
        assert torch.allclose(x, y, rtol=1e-5, atol=1e-7), name
    assert a.host() == b.host()


def test_static_scratch_matches_workspace_entry_point_twice_in_a_row():
    import paper_2609_02780_gb300 as ss
    dev = torch.device("cuda:0")
    keys, q1 = _case(101)
    _, q2 = _case(102)
    P, Hkv, N, _ = keys.shape
    idx = ss.Index(P, 8, Hkv, 40, N // 40, device=dev)
    idx.append(keys.to(dev))
    p = ss.RetrieveParams(k=150, budget=6, n_recent=2)
    uh = N // 40 - 2
    qs = [q1.to(dev), q2.to(dev)]
    refs = []
    for q in qs:
        r = ss.Result(idx, p)
        idx.retrieve(q, k=p.k, budget=p.budget, n_recent=p.n_recent, out=r)
        r.check()
        refs.append(r)
    outs = [ss.Result(idx, p) for _ in range(3)]
    torch.cuda.synchronize()

    def allocations():
        # cumulative count of device allocations made through torch (the binding's
        # allocator too), and the memory torch holds: frees of earlier tests' tensors
        # lower neither
        st = torch.cuda.memory_stats(dev)
        return st["allocation.all.allocated"], torch.cuda.memory_reserved(dev)

    gc.collect()
    gc.disable()
    try:
        before = allocations()
        # two calls in a row on the same question, then a call on another question
        for out, j in zip(outs, (0, 0, 1)):
            idx.retrieve_static(qs[j], p, out)
        torch.cuda.synchronize()
        assert allocations() == before
    finally:
        gc.enable()
    for out, j in zip(outs, (0, 0, 1)):
        out.check()
        _same(out, refs[j], uh)


def test_static_scratch_rejects_a_retrieval_that_does_not_fit():
    import paper_2609_02780_gb300 as ss
    dev = torch.device("cuda:0")
    # 56 lists x ~190k candidate slots x 8 bytes is well above the 64 MiB scratch
    idx = ss.Index(2, 28, 4, 64, 2000, device=dev)
    p = ss.RetrieveParams(k=64, budget=4)
    assert idx.workspace_bytes(4, p) > 64 << 20
    q = torch.zeros(2, 4, 28, 128, dtype=torch.bfloat16, device=dev)
    with pytest.raises(ss.ShallowStreamError, match="CAPACITY"):
        idx.retrieve_static(q, p, ss.Result(idx, p))
