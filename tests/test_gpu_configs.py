"""Parity at the larger configurations (GPU only): the hour-long schedule stress,
the 30-layer Wan-1.3B rollout and the Wan-14B shape.  Every input is synthetic
(AR(1) K/V, N(0,1) Q); the oracle follows sampled coordinates, heads or layers
(merges are elementwise, attention is per head, layers are independent), and the
entry table is compared bit-exactly."""
import numpy as np
import pytest
import torch

from oracle import OracleMemory
from synth import KIND_K, KIND_V, DeviceAR1, device_queries, rho_drift

from parity_utils import BF16_U, Pair, RoundingDepth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module", autouse=True)
def _built(cuda_lib):
    from paper_2606_10671_gb300 import capi
    capi.load(cuda_lib)


def test_hour_long_schedule_stress():
    """12 heads, D=128, N=1560, 1 layer, 20,000 segments (60,000 frames) under a 21-entry
    budget; rho drifts 0.95 -> 0.5.  Checked at 40 checkpoints:
    - the entry table, bit-exact;
    - stored K/V at 4096 fixed sampled coordinates against the oracle.  Each stored value
      is a convex combination of its sources, rounded once per pass that rewrote it, so
      its error is bounded along its merge tree: every rounding adds at most 2^-8 of the
      magnitude of the block it rounds (plus 2^-19 of the sources' for the fp32 weights
      and FMAs), with the exact magnitudes taken from the oracle (RoundingDepth.e); and
      the entry's RMS error stays below 2 sqrt(r) 2^-8 RMS(exact), r its merge depth;
    - at 4 checkpoints, fademem_attend for 64 sampled queries against the oracle's
      attention over the GPU's downloaded memory (heads 0 and 11), at 2e-2."""
    from paper_2606_10671_gb300 import FadeMem
    H, D, N, M, F, SEG = 12, 128, 1560, 21, 3, 20000
    frames_total = F * SEG
    rho = rho_drift(0.95, 0.5, frames_total)
    mem = FadeMem(M, H, D, N, beta=0.3, dtype=torch.bfloat16)
    gk = DeviceAR1((N, H, D), 11, KIND_K, 0, rho)
    gv = DeviceAR1((N, H, D), 11, KIND_V, 0, rho)
    rng = np.random.default_rng(11)
    S = 4096
    n_idx = torch.from_numpy(rng.integers(0, N, S)).cuda()
    h_idx = torch.from_numpy(rng.integers(0, H, S)).cuda()
    d_idx = torch.from_numpy(rng.integers(0, D, S)).cuda()
    ora = OracleMemory(M, 0.3, anchor=True, elems=S)
    chunk = 250
    buf = torch.empty((chunk, F, 2, S), dtype=torch.bfloat16, device="cuda")
    depth = RoundingDepth(anchor=True)  # per entry: depth r and error bound e [K|V][S] along its merge tree
    worst = 0.0
    worst_bound = 0.0
    attn_checks = {4999, 9999, 14999, SEG - 1}
    attn_heads = [0, H - 1]
    q_rows = torch.from_numpy(np.sort(rng.choice(F * N, 64, replace=False))).cuda()
    for seg in range(SEG):
        K = torch.stack([gk.next() for _ in range(F)]).contiguous()
        V = torch.stack([gv.next() for _ in range(F)]).contiguous()
        mem.insert(0, K, V)
        mem.consolidate()
        buf[seg % chunk, :, 0] = K[:, n_idx, h_idx, d_idx]
        buf[seg % chunk, :, 1] = V[:, n_idx, h_idx, d_idx]
        if seg % chunk == chunk - 1 or seg == SEG - 1:
            host = buf.double().cpu().numpy()
            for c in range(seg % chunk + 1):
                _, first, span, _ = ora.entries()
                before = list(zip(first.tolist(), span.tolist()))
                f0 = ora.frames
                fresh = {}
                for f in range(F):
                    ora.insert(host[c, f, 0], host[c, f, 1])
                    fresh[f0 + f] = np.abs(host[c, f])
                _, first, span, _ = ora.entries()
                after = list(zip(first.tolist(), span.tolist()))
                known = set(before)
                exact = {key: np.abs(np.stack(ora.entry_kv(i))) for i, key in enumerate(after) if key not in known}
                depth.update(before, f0, fresh, after, exact=exact)
        if seg % 500 == 499 or seg == SEG - 1:
            assert seg % chunk == chunk - 1 or seg == SEG - 1
            slot, first, span, mu2 = mem.entries()
            o_slot, o_first, o_span, o_mu = ora.entries()
            assert slot.tolist() == o_slot.tolist(), seg
            assert first.tolist() == o_first.tolist(), seg
            assert span.tolist() == o_span.tolist(), seg
            assert mu2.tolist() == [int(round(2 * m)) for m in o_mu], seg
            Kd, Vd = mem.layer_memory(0)
            for i, s in enumerate(slot.tolist()):
                key = (int(first[i]), int(span[i]))
                ko, vo = ora.entry_kv(i)
                kg = Kd[h_idx, s, n_idx, d_idx].double().cpu().numpy()
                vg = Vd[h_idx, s, n_idx, d_idx].double().cpu().numpy()
                r = depth.r[key]
                for kv, (got, ref) in enumerate(((kg, ko), (vg, vo))):
                    err = np.abs(got - ref)
                    bound = depth.e[key][kv] + 1e-12
                    assert np.all(err <= bound), (seg, i, float(err.max()), r)
                    # never looser than the depth x largest-input bound it replaces
                    assert np.all(bound <= r * (BF16_U + 2.0 ** -20) * depth.a[key][kv] * (1 + 2.0 ** -6) + 1e-12)
                    rms, rms_ref = np.sqrt(np.mean(err ** 2)), np.sqrt(np.mean(ref ** 2))
                    assert rms <= 2 * np.sqrt(r) * BF16_U * rms_ref + 1e-12, (seg, i, rms, rms_ref, r)
                    worst = max(worst, float(err.max()))
                    worst_bound = max(worst_bound, float(bound.max()))
        if seg in attn_checks:
            _check_attention_on_downloaded_memory(mem, 0, attn_heads, q_rows, seed=seg)
    assert mem.counts() == (M, frames_total)
    assert span.sum() == frames_total and span.max() > 1000  # merges reach deep into the hierarchy
    mem.device_status()
    print(f"hour-long stress: final spans {span.tolist()}, worst |diff| {worst:.3e}, "
          f"largest per-coordinate bound {worst_bound:.3e}, deepest r {max(depth.r.values())}")


def _check_attention_on_downloaded_memory(mem, layer, heads, rows, seed):
    """fademem_attend of sampled query rows against the oracle's attention over the GPU's
    own stored memory (downloaded; budget above the count, so the oracle merges nothing),
    for the given heads.  The 2e-2 bound then measures the attention kernel alone."""
    c = mem.cfg
    slot = mem.entries()[0]
    Kd, Vd = mem.layer_memory(layer)
    hs = torch.as_tensor(heads, device="cuda")
    ref_mem = OracleMemory(len(slot) + 1, 0.3, elems=c.tokens_per_frame * len(heads) * c.head_dim)
    for s in slot.tolist():  # temporal order
        ref_mem.insert(Kd[hs, s].double().cpu().numpy().transpose(1, 0, 2),
                       Vd[hs, s].double().cpu().numpy().transpose(1, 0, 2))
    Q = device_queries((3 * c.tokens_per_frame, c.heads, c.head_dim), 77, layer, seed)
    out = mem.attend(layer, Q)
    torch.cuda.synchronize()
    ref = ref_mem.attend(Q[rows][:, hs].double().cpu().numpy(), c.tokens_per_frame, len(heads), c.head_dim)
    got = out[rows][:, hs].double().cpu().numpy()
    err = float(np.abs(got - ref).max())
    assert err <= 2e-2, (seed, err)
    return err


def _rollout(layers, heads, segments, check_segments, oracle_layers, tracked_heads, seed):
    """AR rollout: per segment, 4 denoising-step attends on every layer, then insert +
    consolidate once (Sec. 4.1).  The oracle follows `oracle_layers` x `tracked_heads`."""
    p = Pair(21, heads, 128, 1560, beta=0.3, dtype=torch.bfloat16, layers=layers, seed=seed,
             tracked_heads=tracked_heads, device_gen=True, oracle_layers=oracle_layers)
    rng = np.random.default_rng(seed)
    rows = np.unique(np.concatenate([rng.choice(4680, 24, replace=False), [0, 4679]]))
    for seg in range(segments):
        if seg > 0:
            for step in range(4):
                for l in range(layers):
                    Q = p.queries(4680, step=seg * 4 + step, layer=l)
                    if seg in check_segments and step == 3 and l in oracle_layers:
                        p.check_attend(Q, layer=l, rows=rows)
                    else:
                        p.gpu.attend(l, Q)
        p.step(3)
        if seg in check_segments:
            p.check_entries()
            for l in oracle_layers:
                p.check_memory(l)
    p.gpu.device_status()
    return p


def test_wan13b_30_layer_rollout():
    """30 layers, 12 heads, 120 segments x 4 denoising steps, budget 21 (layers 0 and 29,
    heads 0 and 7 followed by the oracle; checks at segments 1, 7, 8, 60 and 119)."""
    _rollout(30, 12, 120, {1, 7, 8, 60, 119}, [0, 29], [0, 7], seed=21)


def test_wan14b_shape():
    """Wan-14B shape: 40 layers, 40 heads, budget 21 (~27 GB of bf16 memory), 60 segments
    x 4 denoising steps; layers 0 and 39, heads 0 and 39 followed; checks at 8, 30, 59."""
    _rollout(40, 40, 60, {8, 30, 59}, [0, 39], [0, 39], seed=14)
