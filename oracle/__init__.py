"""CPU oracle for ShallowStream query-time evidence retrieval.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline (the cpu_baseline leg and the reference arm) may import or run anything in
this package. The product path (the CUDA library and its Python binding) never
imports it and shares no code with it.

Plain, slow, fp64 numpy written from the paper's definitions:
  retrieval.py  Eq. 3 (unit descriptor), Eq. 4 (recent/history split), Sec. 4.2
                scored Q-K attention, Eq. 11 (per-layer top-M), unit votes, the
                vote-ranked pool, max-min diversity, Eq. 12 (temporal expansion)
  kmeans.py     token-level k-means compression of 20-frame windows and retrieval
                over the centroids with member expansion (the cluster-compressed
                index variant; closest paper text Sec. 4.1 Eq. 5-7 and Eq. 13)
  shard.py      one shard's share of a retrieval over an index split by token range
                (its top-k candidates with scores, softmax statistics per list and
                per unit, descriptors)
  unit_clusters.py  the paper's long-history compression (Sec. 4.1, Eq. 5-7: units
                leaving the detailed window clustered online, representative keys as
                running averages) and the cluster evidence of Eq. 13
  forward.py    the question's forward pass through the shallow layers (Eq. 10):
                synthetic pre-norm GQA decoder layers whose attention reads the stored
                keys and values, yielding the query states the retrieval scores
"""
from . import retrieval, kmeans, shard, unit_clusters, forward  # noqa: F401
