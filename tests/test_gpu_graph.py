"""A retrieval captured in a CUDA graph and replayed gives the direct call's results.

Once the result arrays and the workspace exist, the launch sequence needs no
allocation and no host synchronisation and passes every parameter by value, so it can
be captured; replays read the question from the captured input buffer.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu

# whole arrays; the pool, selection, expansion and frames over their valid prefixes
FIELDS = ("topk_tok", "topk_w", "list_stats", "unit_votes", "unit_mass", "counts")


def _same(a, b):
    for f in FIELDS:
        assert torch.equal(getattr(a, f), getattr(b, f)), f
    assert a.host() == b.host()


@pytest.mark.parametrize("head_agg", [0, 1])
def test_graph_replay_matches_direct_calls(head_agg):
    import paper_2609_02780_gb300 as ss
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["tiny"]
    dev = torch.device("cuda:0")
    data = synth.make_workload(w, device=dev)
    idx = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, w.n_frames,
                   device=dev)
    idx.append(data["keys"])
    p = ss.RetrieveParams(k=w.k, budget=w.budget, head_agg=head_agg)
    q_in = data["q"].clone()
    g = torch.Generator(device="cpu").manual_seed(5)
    q_other = torch.randn(q_in.shape, generator=g).to(torch.bfloat16).to(dev)
    ws = torch.empty(idx.workspace_bytes(q_in.shape[1], p), dtype=torch.uint8, device=dev)
    out = ss.Result(idx, p)

    def call(o):
        idx.retrieve(q_in, k=p.k, budget=p.budget, head_agg=p.head_agg, out=o, workspace=ws)

    call(out)                                   # first call outside the capture
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        call(out)
    for q_new in (data["q"], q_other, data["q"]):
        q_in.copy_(q_new)
        graph.replay()
        torch.cuda.synchronize()
        out.check()
        ref = ss.Result(idx, p)
        call(ref)
        ref.check()
        _same(out, ref)
