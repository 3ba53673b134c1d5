"""Host checks of the bookkeeping the GPU parity tests derive their bf16 bounds from
(tests/parity_utils.RoundingDepth), run on the fp64 oracle alone: every entry's exact
block lies within its recorded source magnitude a (merges are convex), new-frame
copies and the anchor are never rounded, and every merged entry's depth r grows by
exactly one per pass over the deepest entry it absorbed."""
import numpy as np

from oracle import OracleMemory
from parity_utils import RoundingDepth


def test_rounding_depth_bounds_every_exact_block():
    M, F, S = 6, 3, 64
    rng = np.random.default_rng(5)
    ora = OracleMemory(M, 0.3, anchor=True, elems=S)
    depth = RoundingDepth(anchor=True)
    deepest = 0
    for seg in range(400):
        _, first, span, _ = ora.entries()
        before = list(zip(first.tolist(), span.tolist()))
        f0 = ora.frames
        fresh = {}
        scale = 1.0 + 4.0 * rng.random()  # magnitudes vary per frame
        for f in range(F):
            K, V = scale * rng.standard_normal(S), scale * rng.standard_normal(S)
            ora.insert(K, V)
            fresh[f0 + f] = np.abs(np.stack([K, V]))
        _, first, span, _ = ora.entries()
        after = list(zip(first.tolist(), span.tolist()))
        depth.update(before, f0, fresh, after)
        assert set(depth.r) == set(after)
        for i, key in enumerate(after):
            ko, vo = ora.entry_kv(i)
            assert np.all(np.abs(np.stack([ko, vo])) <= depth.a[key] * (1 + 1e-15)), (seg, key)
            if key[0] == 0 or (key[1] == 1 and key[0] >= f0):
                assert depth.r[key] == 0, key
            elif key not in before:
                inner = [depth_r for k, depth_r in old_r.items() if k[0] >= key[0] and k[0] + k[1] <= sum(key)]
                assert depth.r[key] == 1 + max(inner, default=0), key
        old_r = dict(depth.r)
        deepest = max(deepest, max(depth.r.values()))
    assert deepest >= 5  # the hierarchy is deep enough for the check to mean something
