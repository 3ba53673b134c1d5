"""bf16 attention with a query tile's keys split over a thread-block cluster (GPU only).

When the (128-query tile, head) CTAs fill less than half the SMs, the launcher
splits each tile's key tiles over a cluster of 2, 4 or 8 CTAs (at least 4 key
tiles each); every CTA keeps its unnormalised (O, m, l) in shared memory and,
after a cluster barrier, assembles a slice of the tile's rows from all of them
through distributed shared memory.  On a 152-SM GB300 these cases take:
  - 2 heads x 1 query tile over 40 key tiles: clusters of 8;
  - 12 heads x 1 query tile over 49 key tiles (the Wan-1.3B head count, one
    128-query tile): clusters of 8, 96 CTAs;
  - one query, one head: clusters of 8, 127 of the tile's rows empty;
  - memory keys and current-chunk keys in the same split (28 + 17 tiles), and
    the chunk's keys alone over an empty memory, and keys re-indexed by temporal RoPE;
  - 3 heads x 3 query tiles (ragged, 300 queries) over 40 tiles: clusters of 8.
Each is checked against the fp64 oracle, and the same call twice gives the same
bytes (the combine adds the CTAs' partials in a fixed order).
"""
import numpy as np
import pytest
import torch

from parity_utils import Pair

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module", autouse=True)
def _built(cuda_lib):
    from paper_2606_10671_gb300 import capi
    capi.load(cuda_lib)


# (budget M, heads H, tokens per frame N, queries Lq, current-chunk keys)
CASES = {
    "two_heads_40_tiles": (5, 2, 1000, 128, 0),
    "twelve_heads_one_tile": (4, 12, 1560, 128, 0),
    "single_query": (5, 1, 1000, 1, 0),
    "memory_and_chunk_keys": (5, 2, 700, 200, 2100),
    "ragged_query_tiles": (5, 3, 1000, 300, 0),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_cluster_split_attention(name):
    M, H, N, Lq, ncur = CASES[name]
    p = Pair(M, H, 128, N, beta=0.3, dtype=torch.bfloat16, seed=57, tracked_heads=list(range(min(H, 3))))
    for seg in range(2):
        p.step(3)
        Q = p.queries(Lq, step=seg)
        if ncur:
            Kc, Vc = p.chunk(ncur, step=seg)
            p.check_attend_ext(Q, Kc, Vc)
            a, b = p.gpu.attend_ext(0, Q, Kc, Vc), p.gpu.attend_ext(0, Q, Kc, Vc)
        else:
            p.check_attend(Q)
            a, b = p.gpu.attend(0, Q), p.gpu.attend(0, Q)
        torch.cuda.synchronize()
        assert torch.equal(a.view(torch.int16), b.view(torch.int16)), "the split attention is not deterministic"
    st, word = p.gpu.device_status()
    assert word == 0


def test_cluster_split_with_temporal_rope():
    """Temporal RoPE (22 pairs): the split attends over the re-indexed keys, 2 heads x 1
    query tile over 40 key tiles (clusters of 8)."""
    p = Pair(5, 2, 128, 1000, beta=0.3, dtype=torch.bfloat16, seed=67, rope_pairs=22)
    for seg in range(3):
        p.step(3)
        p.check_attend(p.queries(128, step=seg))
    st, word = p.gpu.device_status()
    assert word == 0


def test_cluster_split_over_the_chunk_alone():
    """An empty memory: 128 queries of 2 heads attend over the 2100 current-chunk keys
    alone (17 key tiles, clusters of 4 on 152 SMs: at least 4 key tiles a CTA), then with the
    first segment's 17 tiles of memory keys before them (34 tiles, clusters of 8)."""
    p = Pair(5, 2, 128, 700, beta=0.3, dtype=torch.bfloat16, seed=61)
    Q = p.queries(128, step=0)
    Kc, Vc = p.chunk(2100, step=0)
    p.check_attend_ext(Q, Kc, Vc)
    p.step(3)
    p.check_attend_ext(Q, Kc, Vc)
    st, word = p.gpu.device_status()
    assert word == 0


def test_cluster_split_matches_unsplit_launch_shape():
    """The same memory attended by 128 queries (split into clusters) and by 128 copies of
    those queries among 4864 (no split: 38 x 12 tiles fill the GPU): the rows agree within
    the bf16 tolerance of the oracle comparison, sampled against the oracle as well."""
    p = Pair(4, 12, 128, 1560, beta=0.3, dtype=torch.bfloat16, seed=59, tracked_heads=[0, 11])
    for _ in range(2):
        p.step(3)
    Q = p.queries(128, step=3)
    small = p.gpu.attend(0, Q)
    big_q = torch.cat([Q] * 38)
    big = p.gpu.attend(0, big_q)
    torch.cuda.synchronize()
    diff = (small.float() - big[:128].float()).abs().max().item()
    assert diff <= 2e-2, diff
    p.check_attend(big_q, rows=np.array([0, 127, 128 * 37, 128 * 38 - 1]))
    st, word = p.gpu.device_status()
    assert word == 0
