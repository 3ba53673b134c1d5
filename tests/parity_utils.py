"""Drive the CUDA memory (through the C ABI) and the fp64 oracle side by side.

Both sides consume exactly the same inputs: frames drawn by synth/, rounded to
the storage dtype, uploaded for the device and widened to fp64 for the oracle.
No oracle input or expected value is ever taken from the CUDA path.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import OracleMemory
from synth import KIND_K, KIND_V, DeviceAR1, HostAR1, device_queries, host_queries, rho_const

OPS = {"weighted": 0, "average": 1, "select_nearest": 2, "max_pool": 3}

# Tolerances (checked as written here):
#   fp32 outputs and memory: max|gpu - oracle| <= 1e-5 * max|oracle|
#   bf16 attention outputs:  max|gpu - oracle| <= 2e-2 (unit-variance data)
#   bf16 memory contents:    derived from bf16 storage.  A stored block is rewritten
#     (and rounded to nearest even, unit roundoff u = 2^-8) once per consolidation pass
#     that changes it, and every merge is a convex combination, so old errors do not
#     grow: after r roundings along its history, |stored - exact| <= r * u * A, with A
#     the largest |input| so far (no intermediate value exceeds it).  Copies of new
#     frames and the anchor are exact (r = 0).  Also the RMS error of a block must stay
#     below 2 * sqrt(r) * u * RMS(exact), which catches a wrong weight long before the
#     max bound would.
F32_RTOL = 1e-5
BF16_ATOL = 2e-2
BF16_U = 2.0 ** -8


def assert_close(got: np.ndarray, ref: np.ndarray, dtype, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), what
    err = np.max(np.abs(got - ref)) if got.size else 0.0
    if dtype == torch.float32:
        bound = F32_RTOL * max(np.max(np.abs(ref)), 1e-30)
    else:
        bound = BF16_ATOL
    assert err <= bound, f"{what}: max|diff| {err:.3e} > {bound:.3e}"
    return err


class Pair:
    """One FadeMem memory on the GPU and one oracle per layer, fed identical frames."""

    def __init__(self, budget, heads, head_dim, tokens, beta=0.3, anchor=True, op="weighted",
                 dtype=torch.bfloat16, layers=1, seed=0, rho=rho_const(0.9), tracked_heads=None, device_gen=False,
                 oracle_layers=None, rope_pairs=0, rope_theta=10000.0, scale=0.0):
        from paper_2606_10671_gb300 import FadeMem
        self.M, self.H, self.D, self.N, self.L = budget, heads, head_dim, tokens, layers
        self.dtype = dtype
        self.tracked = list(range(heads)) if tracked_heads is None else list(tracked_heads)
        self.gpu = FadeMem(budget, heads, head_dim, tokens, num_layers=layers, beta=beta, anchor=anchor, merge_op=op,
                           dtype=dtype, rope_pairs=rope_pairs, rope_theta=rope_theta, scale=scale)
        self.scale = None if scale == 0.0 else float(scale)  # the oracle's softmax scale (None: 1/sqrt(D))
        self.rope = rope_pairs > 0
        elems = tokens * len(self.tracked) * head_dim
        self.ora_layers = list(range(layers)) if oracle_layers is None else list(oracle_layers)
        self.ora = {l: OracleMemory(budget, beta, anchor=anchor, op=OPS[op], elems=elems) for l in self.ora_layers}
        if rope_pairs:
            for o in self.ora.values():
                o.set_rope(rope_pairs, rope_theta, tokens, len(self.tracked), head_dim)
        shape = (tokens, heads, head_dim)
        if device_gen:
            self.gens = [(DeviceAR1(shape, seed, KIND_K, l, rho, dtype), DeviceAR1(shape, seed, KIND_V, l, rho, dtype))
                         for l in range(layers)]
        else:
            self.gens = [(HostAR1(shape, seed, KIND_K, l, rho), HostAR1(shape, seed, KIND_V, l, rho))
                         for l in range(layers)]
        self.device_gen = device_gen
        self.seed = seed
        self.anchor = anchor
        self.input_max = 0.0
        self.rounds = {}
        self.margins = []  # the oracle's relative margin of every decision, frame by frame

    def _frames(self, gen, n):
        if self.device_gen:
            return torch.stack([gen.next() for _ in range(n)]).contiguous()
        x = np.stack([gen.next() for _ in range(n)])
        return torch.from_numpy(x).to(self.dtype).cuda()

    def insert(self, frames: int, per_call: int | None = None):
        """Insert `frames` frames on every layer (in calls of `per_call` frames), without consolidating."""
        per_call = per_call or frames
        self._keep = []
        for l in range(self.L):
            gk, gv = self.gens[l]
            K = self._frames(gk, frames)
            V = self._frames(gv, frames)
            for a in range(0, frames, per_call):
                b = min(frames, a + per_call)
                self.gpu.insert(l, K[a:b].contiguous(), V[a:b].contiguous())
            self._keep.append((K, V))
            if l not in self.ora:
                continue
            Kt = K[:, :, self.tracked, :].double().cpu().numpy()
            Vt = V[:, :, self.tracked, :].double().cpu().numpy()
            self.input_max = max(self.input_max, float(np.abs(Kt).max()), float(np.abs(Vt).max()))
            for f in range(frames):
                self.ora[l].insert(Kt[f], Vt[f])
                if l == self.ora_layers[0]:
                    self.margins.append(self.ora[l].last_margin)

    def step(self, frames: int = 3, per_call: int | None = None):
        before = self._spans()
        f0 = self._ref().frames
        self.insert(frames, per_call)
        self.gpu.consolidate()
        pc = per_call or frames
        chunks = [min(pc, frames - a) for a in range(0, frames, pc)]
        self._update_rounds(before, f0, sum(-(-c // 4) for c in chunks))  # fused passes of <= 4 frames

    def _ref(self):
        return self.ora[self.ora_layers[0]]

    def _spans(self):
        _, first, span, _ = self._ref().entries()
        return [(int(a), int(s)) for a, s in zip(first, span)]

    def _update_rounds(self, before, frames_before, passes):
        """Rounding depth r of every entry after one consolidate call of `passes` passes."""
        old = {fs: self.rounds.get(fs, 0) for fs in before}
        new = {}
        for a, s in self._spans():
            if (a, s) in old:
                new[(a, s)] = old[(a, s)]
            elif a == 0 and self.anchor:
                new[(a, s)] = 0  # the anchor keeps frame 0's block exactly
            elif s == 1 and a >= frames_before:
                new[(a, s)] = 0  # a copy of a new frame
            else:
                inner = [r for (b, t), r in old.items() if b >= a and b + t <= a + s]
                new[(a, s)] = max(inner, default=0) + passes
        self.rounds = new

    def check_entries(self):
        """The entry table bit-exact against the oracle, and the device status word clear (no
        time-out, count mismatch, plan overflow, uncertified decision or, in the bounds-checking
        build, bounds failure); reading the word clears it."""
        st, word = self.gpu.device_status(raise_on_error=False)
        assert word == 0, f"device status 0x{word:x}"
        slot, first, span, mu2 = self.gpu.entries()
        o_slot, o_first, o_span, o_mu = self._ref().entries()
        assert slot.tolist() == o_slot.tolist(), (slot, o_slot)
        assert first.tolist() == o_first.tolist()
        assert span.tolist() == o_span.tolist()
        assert mu2.tolist() == [int(round(2 * m)) for m in o_mu]
        assert np.all(2 * o_mu == np.round(2 * o_mu))
        return slot

    def check_memory(self, layer=0):
        """Every stored block of every entry, for the tracked heads."""
        Kd, Vd = self.gpu.layer_memory(layer)
        ora = self.ora[layer]
        slot, first, span, _ = ora.entries()
        worst = 0.0
        for i, s in enumerate(slot.tolist()):
            Ko, Vo = ora.entry_kv(i)
            Ko = Ko.reshape(self.N, len(self.tracked), self.D).transpose(1, 0, 2)
            Vo = Vo.reshape(self.N, len(self.tracked), self.D).transpose(1, 0, 2)
            kg = Kd[self.tracked, s].double().cpu().numpy()
            vg = Vd[self.tracked, s].double().cpu().numpy()
            if self.dtype == torch.float32:
                worst = max(worst, assert_close(kg, Ko, self.dtype, f"K entry {i} slot {s}"),
                            assert_close(vg, Vo, self.dtype, f"V entry {i} slot {s}"))
                continue
            r = self.rounds.get((int(first[i]), int(span[i])), 0)
            for got, ref, nm in ((kg, Ko, "K"), (vg, Vo, "V")):
                err = np.abs(got - ref)
                # Temporal RoPE: a stored K block is rotated before its rounding, so even a
                # copy is rounded once, and rotated components reach sqrt(2) * A.  (The
                # anchor's frame 0 rotates by 0 and stays exact, within this bound.)
                rk, amax = (max(r, 1), np.sqrt(2.0) * self.input_max) if self.rope and nm == "K" \
                    else (r, self.input_max)
                bound = rk * (BF16_U + 2.0 ** -20) * amax + 1e-12  # + fp32 accumulation
                r_rms = rk
                assert np.all(np.isfinite(got)), nm
                assert err.max() <= bound, f"{nm} entry {i} slot {s}: max|diff| {err.max():.3e} > {bound:.3e} (r={r})"
                rms = np.sqrt(np.mean(err ** 2))
                assert rms <= 2 * np.sqrt(r_rms) * BF16_U * np.sqrt(np.mean(ref ** 2)) + 1e-12, \
                    f"{nm} entry {i} slot {s}: rms diff {rms:.3e} (r={r_rms})"
                worst = max(worst, float(err.max()))
        return worst

    def queries(self, Lq, step=0, layer=0):
        if self.device_gen:
            return device_queries((Lq, self.H, self.D), self.seed, layer, step, dtype=self.dtype)
        q = host_queries((Lq, self.H, self.D), self.seed, layer, step)
        return torch.from_numpy(q).to(self.dtype).cuda()

    def chunk(self, ncur, step=0, layer=0):
        """Keys and values of a current chunk [ncur, H, D] (its own stream, N(0,1))."""
        g = np.random.default_rng([self.seed, 77, layer, step])
        K = g.standard_normal((ncur, self.H, self.D), dtype=np.float32)
        V = g.standard_normal((ncur, self.H, self.D), dtype=np.float32)
        return torch.from_numpy(K).to(self.dtype).cuda(), torch.from_numpy(V).to(self.dtype).cuda()

    def check_attend_ext(self, Q: torch.Tensor, Kcur: torch.Tensor, Vcur: torch.Tensor, layer=0, rows=None):
        out = self.gpu.attend_ext(layer, Q, Kcur, Vcur)
        torch.cuda.synchronize()
        if rows is not None:
            idx = torch.as_tensor(np.asarray(rows), device=Q.device)
            Q, out = Q[idx], out[idx]
        Qt = Q.double().cpu().numpy()[:, self.tracked, :]
        Kc = Kcur.double().cpu().numpy()[:, self.tracked, :]
        Vc = Vcur.double().cpu().numpy()[:, self.tracked, :]
        ref = self.ora[layer].attend_ext(Qt, Kc, Vc, self.N, len(self.tracked), self.D, scale=self.scale)
        return assert_close(out.double().cpu().numpy()[:, self.tracked, :], ref, self.dtype, "attention + chunk")

    def check_attend(self, Q: torch.Tensor, layer=0, rows=None):
        out = self.gpu.attend(layer, Q)
        torch.cuda.synchronize()
        if rows is not None:
            idx = torch.as_tensor(np.asarray(rows), device=Q.device)
            Q, out = Q[idx], out[idx]
        Qh = Q.double().cpu().numpy()
        og = out.double().cpu().numpy()
        Qt = Qh[:, self.tracked, :]
        ref = self.ora[layer].attend(Qt, self.N, len(self.tracked), self.D, scale=self.scale)
        return assert_close(og[:, self.tracked, :], ref, self.dtype, "attention")


class RoundingDepth:
    """Bookkeeping of bf16 storage rounding per memory entry, keyed by (first, span).

    r: the number of consolidation passes that rewrote (and so rounded) the entry's
    block along its history (its deepest chain of merges); copies of new frames and
    the anchor have r = 0.  a: the largest |input| over the entry's own source frames,
    per coordinate.  Merges are convex and elementwise, so the exact block and every
    rounded intermediate lie within +-a, and |stored - exact| <= r (2^-8 + 2^-20) a.

    e (when the exact new blocks are given, one pass per call): a tighter bound per
    coordinate, built along the merge tree.  A pass writes each merged entry as
    round_bf16(sum_k w_k stored_k) over its sources k (the older entries it covers
    and the new frames in its span), with fp32 weights and fp32 FMAs.  With
    stored_k = exact_k + err_k, |err_k| <= e_k, convex weights and x = |exact|:
      before rounding:  |y - exact_new| <= E = max_k e_k + 2^-19 max_k (x_k + e_k)
                        (2^-20 for the fp32 weights, 2^-20 for the FMA chain);
      after rounding:   e_new = E + 2^-8 (x_new + E).
    Each rounding then costs 2^-8 of the magnitude of the block it rounds, not of
    the largest input, which is what makes deep merged entries checkable.
    """

    def __init__(self, anchor: bool = True):
        self.anchor = anchor
        self.r = {}
        self.a = {}
        self.e = {}
        self.x = {}
        self.anchor_a = None

    def update(self, before, frames_before, fresh, after, passes: int = 1, exact=None):
        """One consolidate call: `before`/`after` the (first, span) lists of the entries,
        `fresh` {frame: |values|} of the frames it inserted, `passes` fused passes,
        `exact` {(first, span): |exact block|} of the entries it created (optional)."""
        if 0 in fresh:
            self.anchor_a = fresh[0]
        old = set(before)
        r, a, e, x = {}, {}, {}, {}
        for key in after:
            f, s = key
            if key in old:
                r[key], a[key] = self.r[key], self.a[key]
                if key in self.e:
                    e[key], x[key] = self.e[key], self.x[key]
            elif f == 0 and self.anchor:
                r[key], a[key] = 0, self.anchor_a
                e[key], x[key] = np.zeros_like(self.anchor_a), self.anchor_a
            elif s == 1 and f >= frames_before:
                r[key], a[key] = 0, fresh[f]
                e[key], x[key] = np.zeros_like(fresh[f]), fresh[f]
            else:
                inner = [k for k in self.r if k[0] >= f and k[0] + k[1] <= f + s]
                new_frames = [v for g, v in fresh.items() if f <= g < f + s]
                parts = [self.a[k] for k in inner] + new_frames
                r[key] = passes + max([self.r[k] for k in inner], default=0)
                a[key] = np.maximum.reduce(parts)
                if exact is not None and passes == 1 and all(k in self.e for k in inner):
                    zero = np.zeros_like(a[key])
                    emax = np.maximum.reduce([self.e[k] for k in inner] + [zero])
                    src = np.maximum.reduce([self.x[k] + self.e[k] for k in inner] + new_frames)
                    pre = emax + 2.0 ** -19 * src
                    x[key] = exact[key]
                    e[key] = pre + BF16_U * (exact[key] + pre)
        self.r, self.a, self.e, self.x = r, a, e, x
