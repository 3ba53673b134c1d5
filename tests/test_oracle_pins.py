"""Pins of the fp64 oracle against what the paper and mathematics fix (CPU only).

Each test ties one part of the oracle to something other than the oracle:
hand-derived worked examples of Algorithm S1, the exact integer schedule at
beta = 1, a 40-digit decimal re-evaluation of the warped gaps, the invariants
of adjacency-only merging (Sec. 3.3), closed-form merge weights, and plain
softmax attention computed by numpy.
"""
import math
import os
from decimal import Decimal, getcontext
from fractions import Fraction

import numpy as np
import pytest

from oracle import OracleMemory, OP_AVERAGE, OP_MAX_POOL, OP_SELECT_NEAREST, OP_WEIGHTED

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name, with_gmin=False):
    rows = []
    with open(os.path.join(GOLDEN, name)) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            parts = line.split()
            t, j = int(parts[0]), int(parts[1])
            gmin = float(parts[2]) if with_gmin else None
            ents = [tuple(p.split(":")) for p in parts[3 if with_gmin else 2:]]
            ents = [(int(a), int(b), int(c), float(d)) for a, b, c, d in ents]
            rows.append((t, j, gmin, ents))
    return rows


def _state(mem):
    slot, first, span, mu = mem.entries()
    return [(int(a), int(b), int(c), float(d)) for a, b, c, d in zip(slot, first, span, mu)]


@pytest.mark.parametrize("name,beta,anchor,with_gmin", [
    ("alg_s1_M4_beta1_anchor.txt", 1.0, True, False),
    ("alg_s1_M4_beta0.3_anchor.txt", 0.3, True, True),
    ("alg_s1_M4_beta1_noanchor.txt", 1.0, False, False),
])
def test_worked_examples(name, beta, anchor, with_gmin):
    """Algorithm S1 step by step against hand-derived states (tests/golden)."""
    rows = {r[0]: r for r in _read_golden(name, with_gmin)}
    mem = OracleMemory(4, beta, anchor=anchor)
    for t in range(10):
        j = mem.insert()
        if t in rows:
            _, j_ref, gmin_ref, ents = rows[t]
            assert j == j_ref, (t, j, j_ref)
            assert _state(mem) == ents, (t, _state(mem), ents)
            if gmin_ref is not None:
                assert abs(mem.last_gmin - gmin_ref) < 1e-4


def _check_invariants(mem, M, anchor):
    slot, first, span, mu = mem.entries()
    n = mem.count
    t = mem.frames - 1
    assert n == min(mem.frames, M)                       # |M_t| <= M, one merge per overflow
    assert span.sum() == mem.frames                      # spans cover the whole history
    assert first[0] == 0
    assert np.all(first[1:] == first[:-1] + span[:-1])   # contiguous, ordered (adjacent merges only)
    assert span[-1] == 1 and first[-1] == t              # newest entry is protected
    assert sorted(slot.tolist()) == list(range(n))       # slot table is a permutation
    assert np.all(np.diff(mu) > 0)                       # temporal order
    mid = first + (span - 1) / 2.0                       # span-weighted centre of a contiguous run
    if anchor:
        assert mu[0] == 0.0
        assert np.all(mu[1:] == mid[1:])
    else:
        assert np.all(mu == mid)


@pytest.mark.parametrize("M,beta,anchor,frames", [
    (8, 0.3, True, 36), (21, 0.3, True, 360), (21, 0.3, True, 60000), (4, 1.0, True, 500),
    (12, 0.5, False, 2000), (21, 0.9, True, 3000), (2, 0.3, True, 50), (3, 0.1, False, 300),
])
def test_invariants(M, beta, anchor, frames):
    """Budget, tiling of the history, ordering, mu = midpoint, every step."""
    mem = OracleMemory(M, beta, anchor=anchor)
    stride = 1 if frames <= 5000 else 97
    for t in range(frames):
        mem.insert()
        if t % stride == 0 or t == frames - 1:
            _check_invariants(mem, M, anchor)


def _closed_form_j_beta1(first, span, anchor):
    """beta = 1: g_i = mu_{i+1} - mu_i, integer/half-integer, from spans alone."""
    mu = [Fraction(int(a)) + Fraction(int(s) - 1, 2) for a, s in zip(first, span)]
    if anchor:
        mu[0] = Fraction(0)
    n = len(mu)
    g = [mu[i + 1] - mu[i] for i in range(n - 2)]
    return min(range(len(g)), key=lambda i: (g[i], i))


@pytest.mark.parametrize("M,anchor", [(4, True), (6, True), (21, True), (5, False), (21, False)])
def test_beta1_exact_schedule(M, anchor):
    """At beta = 1 every gap is exact; ties everywhere exercise the lowest-index rule."""
    mem = OracleMemory(M, 1.0, anchor=anchor)
    for t in range(2000):
        before = None
        if mem.count == M:
            _, first, span, _ = mem.entries()
            first = list(first) + [t]
            span = list(span) + [1]
            before = _closed_form_j_beta1(first, span, anchor)
        j = mem.insert()
        if before is not None:
            assert j == before, t


def _decimal_pow(x, beta):
    return Decimal(x) ** Decimal(beta)


def _exact_schedule(M, beta, frames, anchor):
    """Independent exact re-simulation of the schedule: rational centres, 40-digit
    decimal gaps.  Returns the chosen pair per frame, the final entries and the
    smallest relative margin between the best and second-best gap."""
    getcontext().prec = 40
    ents = []  # [first, span, mu as Fraction]
    js, worst = [], 1.0
    for t in range(frames):
        ents.append([t, 1, Fraction(t)])
        j_ref = -1
        if len(ents) > M:
            g = []
            for i in range(len(ents) - 2):
                di = Fraction(t) - ents[i][2]
                di1 = Fraction(t) - ents[i + 1][2]
                ui = _decimal_pow(Decimal(di.numerator) / Decimal(di.denominator), beta)
                ui1 = _decimal_pow(Decimal(di1.numerator) / Decimal(di1.denominator), beta)
                g.append(abs(ui1 - ui))
            j_ref = min(range(len(g)), key=lambda i: (g[i], i))
            if len(g) > 1:
                srt = sorted(g)
                worst = min(worst, float((srt[1] - srt[0]) / srt[1]))
            a, b = ents[j_ref], ents[j_ref + 1]
            s = a[1] + b[1]
            mu = Fraction(0) if (anchor and j_ref == 0) else (a[1] * a[2] + b[1] * b[2]) / s
            ents[j_ref:j_ref + 2] = [[a[0], s, mu]]
        js.append(j_ref)
    return js, ents, worst


@pytest.mark.parametrize("M,beta,frames,anchor,ties", [(21, "0.3", 360, True, False), (8, "0.3", 36, True, False),
                                                       (6, "0.5", 200, False, True), (21, "0.7", 300, True, False)])
def test_decimal_schedule(M, beta, frames, anchor, ties):
    """fp64 oracle vs an exact re-simulation (40-digit gaps, rational centres):
    same pair at every frame and same final state.  At beta=0.3/0.7 every argmin
    also wins by a clear margin; at beta=0.5 perfect squares give exact ties
    (sqrt9 - sqrt4 = sqrt4 - sqrt1), which the lowest-index rule settles."""
    js, ents, worst = _exact_schedule(M, beta, frames, anchor)
    mem = OracleMemory(M, float(beta), anchor=anchor)
    for t in range(frames):
        assert mem.insert() == js[t], t
    _, first, span, mu = mem.entries()
    assert [e[0] for e in ents] == first.tolist()
    assert [e[1] for e in ents] == span.tolist()
    assert [float(e[2]) for e in ents] == mu.tolist()
    if ties:
        assert worst == 0.0
    else:
        assert worst > 1e-9


@pytest.mark.parametrize("M,beta,frames,rho_drift", [(21, 0.3, 60000, True), (21, 0.3, 360, False),
                                                     (8, 0.3, 36, False)])
def test_no_near_ties(M, beta, frames, rho_drift):
    """Certificate used by the device parity: every fp64 argmin at beta=0.3 wins by a
    relative margin far above fp64 rounding (so any pow within a few ulp agrees)."""
    mem = OracleMemory(M, beta, anchor=True)
    worst = 1.0
    for _ in range(frames):
        mem.insert()
        if mem.last_margin < math.inf:
            worst = min(worst, mem.last_margin)
    assert worst > 1e-9, worst


def _run_blocks(M, beta, anchor, op, blocks):
    mem = OracleMemory(M, beta, anchor=anchor, op=op, elems=blocks[0][0].size)
    for K, V in blocks:
        mem.insert(K, V)
    return mem


def test_merge_weights_closed_form():
    """Square-root span weights on the M=4, beta=1 example (Sec. 3.3 operator).

    After t=8 the entries hold frames {0,1}, {2,3}, {4..7}, {8}; their K blocks
    must be: frame 0 (anchor, bit-identical), (c2+c3)/2 (equal spans -> plain
    average), and for {4..7}: merge of {4,5} (average) with 6 at weights
    (2-sqrt2, sqrt2-1) [= sqrt2/(sqrt2+1)], then with 7 at ((3-sqrt3)/2, (sqrt3-1)/2).
    """
    rng = np.random.default_rng(5)
    c = [rng.standard_normal(16) for _ in range(9)]
    blocks = [(c[t], -c[t]) for t in range(9)]
    mem = _run_blocks(4, 1.0, True, OP_WEIGHTED, blocks)
    K0, V0 = mem.entry_kv(0)
    assert np.array_equal(K0, c[0]) and np.array_equal(V0, -c[0])
    K1, _ = mem.entry_kv(1)
    np.testing.assert_allclose(K1, (c[2] + c[3]) / 2, rtol=0, atol=1e-15)
    K2, V2 = mem.entry_kv(2)
    w45 = (c[4] + c[5]) / 2
    r2 = math.sqrt(2.0)
    k456 = (2 - r2) * w45 + (r2 - 1) * c[6]
    r3 = math.sqrt(3.0)
    expect = (3 - r3) / 2 * k456 + (r3 - 1) / 2 * c[7]
    np.testing.assert_allclose(K2, expect, rtol=0, atol=1e-14)
    np.testing.assert_allclose(V2, -expect, rtol=0, atol=1e-14)
    K3, _ = mem.entry_kv(3)
    assert np.array_equal(K3, c[8])


def test_merge_operator_properties():
    """Convexity, idempotence on identical blocks, and the ablation operators (Table 2)."""
    rng = np.random.default_rng(7)
    blocks = [(rng.standard_normal(32), rng.standard_normal(32)) for _ in range(40)]
    for op in (OP_WEIGHTED, OP_AVERAGE, OP_SELECT_NEAREST):
        mem = _run_blocks(5, 0.3, True, op, blocks)
        lo = np.min([b[0] for b in blocks], axis=0)
        hi = np.max([b[0] for b in blocks], axis=0)
        for i in range(mem.count):
            K, _ = mem.entry_kv(i)
            assert np.all(K >= lo - 1e-12) and np.all(K <= hi + 1e-12)
    same = [(np.full(8, 1.25), np.full(8, -0.5))] * 30
    mem = _run_blocks(4, 0.3, False, OP_WEIGHTED, same)
    for i in range(mem.count):
        K, V = mem.entry_kv(i)
        np.testing.assert_allclose(K, 1.25, atol=1e-15)
        np.testing.assert_allclose(V, -0.5, atol=1e-15)
    # Average: two unit-span entries merge to their plain mean (M=2: t=2 merges frames 0,1 w/o anchor).
    b = [(np.array([1.0, 4.0]), np.array([0.0, 2.0])), (np.array([3.0, -2.0]), np.array([2.0, 2.0])),
         (np.array([9.0, 9.0]), np.array([9.0, 9.0]))]
    mem = _run_blocks(2, 0.3, False, OP_AVERAGE, b)
    np.testing.assert_array_equal(mem.entry_kv(0)[0], [2.0, 1.0])
    mem = _run_blocks(2, 0.3, False, OP_SELECT_NEAREST, b)
    np.testing.assert_array_equal(mem.entry_kv(0)[0], [3.0, -2.0])
    mem = _run_blocks(2, 0.3, False, OP_MAX_POOL, b)
    np.testing.assert_array_equal(mem.entry_kv(0)[0], [3.0, 4.0])
    np.testing.assert_array_equal(mem.entry_kv(0)[1], [2.0, 2.0])


def _numpy_attention(Q, Kall, Vall, scale):
    """Plain softmax attention per head (numpy fp64; independent of the oracle)."""
    from scipy.special import softmax
    logits = np.einsum("qhd,khd->hqk", Q, Kall) * scale
    p = softmax(logits, axis=-1)
    return np.einsum("hqk,khd->qhd", p, Vall)


def test_attention_no_merge_equals_full_attention():
    """Budget >= history: no merges, so the output is full attention over all frames."""
    rng = np.random.default_rng(11)
    N, H, D, F = 5, 3, 8, 6
    frames = [(rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D))) for _ in range(F)]
    mem = OracleMemory(8, 0.3, anchor=True, elems=N * H * D)
    for K, V in frames:
        mem.insert(K, V)
    Q = rng.standard_normal((7, H, D)) * 2.0
    out = mem.attend(Q, N, H, D)
    Kall = np.concatenate([f[0] for f in frames])
    Vall = np.concatenate([f[1] for f in frames])
    ref = _numpy_attention(Q, Kall, Vall, 1 / math.sqrt(D))
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-13)
    out2 = mem.attend(Q, N, H, D, scale=0.37)
    np.testing.assert_allclose(out2, _numpy_attention(Q, Kall, Vall, 0.37), rtol=1e-12, atol=1e-13)


def test_attention_special_cases():
    """One key: out = v.  Zero queries: the mean of every cached value row."""
    rng = np.random.default_rng(3)
    H, D = 2, 4
    K, V = rng.standard_normal((1, H, D)), rng.standard_normal((1, H, D))
    mem = OracleMemory(4, 0.3, elems=H * D)
    mem.insert(K, V)
    out = mem.attend(rng.standard_normal((3, H, D)) * 10, 1, H, D)
    np.testing.assert_allclose(out, np.broadcast_to(V, (3, H, D)), rtol=0, atol=1e-15)
    N = 6
    mem = OracleMemory(3, 0.3, elems=N * H * D)
    vals = []
    for _ in range(7):  # 7 frames through a 3-entry budget: merges happen
        K, V = rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D))
        mem.insert(K, V)
    for i in range(mem.count):
        vals.append(mem.entry_kv(i)[1].reshape(N, H, D))
    out = mem.attend(np.zeros((2, H, D)), N, H, D)
    ref = np.concatenate(vals).mean(axis=0)
    np.testing.assert_allclose(out, np.broadcast_to(ref, (2, H, D)), rtol=0, atol=1e-14)


def test_attention_after_merges_uses_merged_blocks():
    """With merges, attention runs over the consolidated entries (numpy on the oracle's blocks)."""
    rng = np.random.default_rng(13)
    N, H, D = 4, 2, 8
    mem = OracleMemory(4, 0.3, anchor=True, elems=N * H * D)
    for _ in range(11):
        mem.insert(rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D)))
    Ks, Vs = zip(*[mem.entry_kv(i) for i in range(mem.count)])
    Kall = np.concatenate([k.reshape(N, H, D) for k in Ks])
    Vall = np.concatenate([v.reshape(N, H, D) for v in Vs])
    Q = rng.standard_normal((5, H, D))
    np.testing.assert_allclose(mem.attend(Q, N, H, D), _numpy_attention(Q, Kall, Vall, 1 / math.sqrt(D)),
                               rtol=1e-12, atol=1e-13)


def test_oracle_rejects_bad_arguments():
    with pytest.raises(ValueError):
        OracleMemory(1, 0.3)
    with pytest.raises(ValueError):
        OracleMemory(4, 0.0)
    with pytest.raises(ValueError):
        OracleMemory(4, 1.5)


def test_attention_with_current_chunk_equals_full_attention():
    """Memory plus current chunk (the paper's cached entries + the chunk's own frames):
    with no merges it is full attention over every frame followed by the chunk; with an
    empty memory it is attention over the chunk alone; with no chunk it is attend()."""
    rng = np.random.default_rng(17)
    N, H, D, F, C = 4, 2, 8, 5, 7
    frames = [(rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D))) for _ in range(F)]
    Kc, Vc = rng.standard_normal((C, H, D)), rng.standard_normal((C, H, D))
    Q = rng.standard_normal((6, H, D))
    mem = OracleMemory(8, 0.3, elems=N * H * D)
    empty = OracleMemory(8, 0.3, elems=N * H * D)
    np.testing.assert_allclose(empty.attend_ext(Q, Kc, Vc, N, H, D), _numpy_attention(Q, Kc, Vc, 1 / math.sqrt(D)),
                               rtol=1e-12, atol=1e-13)
    for K, V in frames:
        mem.insert(K, V)
    Kall = np.concatenate([f[0] for f in frames] + [Kc])
    Vall = np.concatenate([f[1] for f in frames] + [Vc])
    np.testing.assert_allclose(mem.attend_ext(Q, Kc, Vc, N, H, D), _numpy_attention(Q, Kall, Vall, 1 / math.sqrt(D)),
                               rtol=1e-12, atol=1e-13)
    none = np.zeros((0, H, D))
    np.testing.assert_array_equal(mem.attend_ext(Q, none, none, N, H, D), mem.attend(Q, N, H, D))


# ---- temporal RoPE (Sec. 3.3, "Boundary and positional handling") ----------------
# The model's keys carry RoPE: pair k = (dims 2k, 2k+1) read as the complex number
# x + iy is multiplied by exp(i * position * theta^(-2k/d)), d = 2P real dims in the
# temporal band (Su et al., RoFormer, Eq. 13-15).  These tests build such keys with
# numpy complex arithmetic, independently of the oracle's own rotation code.

def _rope(X, position, pairs, theta):
    """Apply RoPE at `position` to the first `pairs` complex pairs of the last axis of X."""
    X = np.array(X, dtype=np.float64, copy=True)
    k = np.arange(pairs)
    z = X[..., 0:2 * pairs:2] + 1j * X[..., 1:2 * pairs:2]
    z = z * np.exp(1j * position * theta ** (-2.0 * k / (2 * pairs)))
    X[..., 0:2 * pairs:2] = z.real
    X[..., 1:2 * pairs:2] = z.imag
    return X


def test_rope_stored_keys_are_phase_free():
    """A key the model rotated to its frame's position t is stored exactly as the
    unrotated key, whatever t; dims outside the temporal band and values are untouched."""
    rng = np.random.default_rng(41)
    N, H, D, P, theta = 3, 2, 16, 5, 10000.0
    mem = OracleMemory(8, 0.3, elems=N * H * D)
    mem.set_rope(P, theta, N, H, D)
    raw = []
    for t in range(6):
        k0, v = rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D))
        raw.append((k0, v))
        mem.insert(_rope(k0, t, P, theta), v)
    for i, (k0, v) in enumerate(raw):
        K, V = mem.entry_kv(i)
        np.testing.assert_allclose(K.reshape(N, H, D), k0, rtol=0, atol=1e-12)
        np.testing.assert_array_equal(V.reshape(N, H, D), v)


def test_rope_without_merges_restores_true_positions():
    """Budget >= history: re-indexing puts entry i at position t_next - count + i = i,
    its own frame, so attention over the memory equals attention over the model's own
    RoPE keys (plain attention, pinned above against numpy)."""
    rng = np.random.default_rng(42)
    N, H, D, P, theta, F = 4, 2, 16, 6, 500.0, 5
    mem = OracleMemory(8, 0.3, elems=N * H * D)
    mem.set_rope(P, theta, N, H, D)
    keys, vals = [], []
    for t in range(F):
        k = _rope(rng.standard_normal((N, H, D)), t, P, theta)
        v = rng.standard_normal((N, H, D))
        keys.append(k)
        vals.append(v)
        mem.insert(k, v)
    Q = _rope(rng.standard_normal((7, H, D)), F, P, theta)
    out = mem.attend(Q, N, H, D)
    ref = _numpy_attention(Q, np.concatenate(keys), np.concatenate(vals), 1 / math.sqrt(D))
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)
    Kc = _rope(rng.standard_normal((3, H, D)), F, P, theta)
    Vc = rng.standard_normal((3, H, D))
    out = mem.attend_ext(Q, Kc, Vc, N, H, D)
    ref = _numpy_attention(Q, np.concatenate(keys + [Kc]), np.concatenate(vals + [Vc]), 1 / math.sqrt(D))
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)


def test_rope_reindex_after_eviction():
    """Budget 2 with the anchor: every pass merges the anchor pair and keeps frame 0's
    block (Algorithm S1), so after frames 0..3 the memory is [frame 0, frame 3].  Re-indexed
    to positions 2 and 3 (right before the query chunk at 4), the attention keys are frame
    0's raw key at position 2 and frame 3's at its own position 3."""
    rng = np.random.default_rng(43)
    N, H, D, P, theta = 2, 1, 8, 3, 100.0
    mem = OracleMemory(2, 0.5, anchor=True, elems=N * H * D)
    mem.set_rope(P, theta, N, H, D)
    raw = [(rng.standard_normal((N, H, D)), rng.standard_normal((N, H, D))) for _ in range(4)]
    for t, (k0, v) in enumerate(raw):
        mem.insert(_rope(k0, t, P, theta), v)
    slot, first, span, mu = mem.entries()
    assert list(first) == [0, 3] and list(span) == [3, 1]
    Q = _rope(rng.standard_normal((5, H, D)), 4, P, theta)
    out = mem.attend(Q, N, H, D)
    Kref = np.concatenate([_rope(raw[0][0], 2, P, theta), _rope(raw[3][0], 3, P, theta)])
    Vref = np.concatenate([raw[0][1], raw[3][1]])
    np.testing.assert_allclose(out, _numpy_attention(Q, Kref, Vref, 1 / math.sqrt(D)), rtol=1e-11, atol=1e-12)
    # A wrong direction or offset is caught: position 1 for frame 0 gives other outputs.
    Kbad = np.concatenate([_rope(raw[0][0], 1, P, theta), _rope(raw[3][0], 3, P, theta)])
    assert np.max(np.abs(out - _numpy_attention(Q, Kbad, Vref, 1 / math.sqrt(D)))) > 1e-6


def test_rope_rejects_bad_arguments():
    mem = OracleMemory(4, 0.3, elems=2 * 1 * 8)
    for bad in ((0, 1e4, 2, 1, 8), (5, 1e4, 2, 1, 8), (2, 1.0, 2, 1, 8), (2, 1e4, 3, 1, 8)):
        with pytest.raises(ValueError):
            mem.set_rope(*bad)
    mem.insert(np.zeros(16), np.zeros(16))
    with pytest.raises(ValueError):
        mem.set_rope(2, 1e4, 2, 1, 8)
