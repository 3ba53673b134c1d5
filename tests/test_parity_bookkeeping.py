"""Host checks of the bookkeeping the GPU parity tests derive their bf16 bounds from
(tests/parity_utils.RoundingDepth), run on the fp64 oracle alone: every entry's exact
block lies within its recorded source magnitude a (merges are convex), new-frame
copies and the anchor are never rounded, every merged entry's depth r grows by
exactly one per pass over the deepest entry it absorbed, and the merge-tree bound e
is zero for unrounded blocks, at least one rounding of the block itself for merged
ones, grows with the bounds it absorbs and is never looser than r (2^-8 + 2^-20) a."""
import numpy as np

from oracle import OracleMemory
from parity_utils import BF16_U, RoundingDepth


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
        exact = {key: np.abs(np.stack(ora.entry_kv(i))) for i, key in enumerate(after) if key not in before}
        old_e = dict(depth.e)
        depth.update(before, f0, fresh, after, exact=exact)
        assert set(depth.r) == set(after)
        for i, key in enumerate(after):
            ko, vo = ora.entry_kv(i)
            assert np.all(np.abs(np.stack([ko, vo])) <= depth.a[key] * (1 + 1e-15)), (seg, key)
            e = depth.e[key]
            assert np.all(e >= 0) and np.all(e <= depth.r[key] * (BF16_U + 2.0 ** -20) * depth.a[key] * (1 + 2.0 ** -6))
            if key[0] == 0 or (key[1] == 1 and key[0] >= f0):
                assert depth.r[key] == 0, key
                assert np.all(e == 0), key
            elif key not in before:
                inner = [depth_r for k, depth_r in old_r.items() if k[0] >= key[0] and k[0] + k[1] <= sum(key)]
                assert depth.r[key] == 1 + max(inner, default=0), key
                assert np.all(e >= BF16_U * exact[key]), key  # the block's own rounding
                absorbed = [old_e[k] for k in old_r if k[0] >= key[0] and k[0] + k[1] <= sum(key)]
                assert all(np.all(e >= x) for x in absorbed), key
        old_r = dict(depth.r)
        deepest = max(deepest, max(depth.r.values()))
    assert deepest >= 5  # the hierarchy is deep enough for the check to mean something


def _bf16(x):
    """Round to the nearest bf16 (ties to even), through fp32."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def test_merge_tree_bound_holds_for_a_rounded_memory():
    """An emulated bf16 memory stays within RoundingDepth.e of the exact one.  The
    emulator follows the oracle's decisions frame by frame (the merged pair read off
    its entry lists), merges blocks with the sqrt-span weights of Sec. 3.3 in fp64,
    keeps the anchor's block, and rounds each merged block to bf16 once per 3-frame
    pass, as the device does (inputs are bf16 values, so copies are exact)."""
    M, F, S = 6, 3, 256
    rng = np.random.default_rng(9)
    ora = OracleMemory(M, 0.3, anchor=True, elems=S)
    depth = RoundingDepth(anchor=True)
    emu = []  # [(first, span, block [2][S])] in temporal order
    worst = 0.0
    for seg in range(300):
        _, first, span, _ = ora.entries()
        before = list(zip(first.tolist(), span.tolist()))
        f0 = ora.frames
        fresh, changed = {}, set()
        scale = 1.0 + 4.0 * rng.random()
        for f in range(F):
            blk = _bf16(scale * rng.standard_normal((2, S)))
            ora.insert(blk[0], blk[1])
            fresh[f0 + f] = np.abs(blk)
            emu.append((f0 + f, 1, blk))
            _, first, span, _ = ora.entries()
            now = list(zip(first.tolist(), span.tolist()))
            if len(now) == len(emu):
                continue
            j = next(i for i in range(len(now)) if now[i] != emu[i][:2])  # the merged pair (j, j + 1)
            (fa, sa, ba), (_, sb, bb) = emu[j], emu[j + 1]
            assert now[j] == (fa, sa + sb)
            if fa == 0:
                blk_new = ba  # the anchor keeps its block
            else:
                wa = np.sqrt(sa) / (np.sqrt(sa) + np.sqrt(sb))
                blk_new = wa * ba + (1.0 - wa) * bb
                changed.add(now[j])
            emu[j:j + 2] = [(fa, sa + sb, blk_new)]
        after = list(zip(first.tolist(), span.tolist()))
        emu = [(a, s, _bf16(b) if (a, s) in changed else b) for a, s, b in emu]  # one rounding per pass
        exact = {key: np.abs(np.stack(ora.entry_kv(i))) for i, key in enumerate(after) if key not in before}
        depth.update(before, f0, fresh, after, exact=exact)
        for i, (a, s, b) in enumerate(emu):
            err = np.abs(b - np.stack(ora.entry_kv(i)))
            assert np.all(err <= depth.e[(a, s)] + 1e-12), (seg, (a, s), float(err.max()))
            worst = max(worst, float((err / (depth.e[(a, s)] + 1e-30)).max()))
    assert worst > 0.05  # the bound is not vacuous: some error comes within 20x of it
