"""fademem_consolidate_noalloc against fademem_consolidate (GPU only).

The allocation-free entry point serves callers that may not allocate device
memory while they run (plug-ins of a host framework that owns all device
memory, real-time loops that fix their memory at start-up): its per-call
working state lives in a static device array of the library.  Through the C
ABI, two memories fed the same frames, one consolidated by each entry point,
must hold the same entry table and the same K/V blocks, and attend the same,
on consecutive calls.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

from synth import KIND_K, KIND_V, HostAR1, host_queries

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

F32_RTOL = 1e-5   # the parity tests' tolerances
BF16_ATOL = 2e-2


def _close(a: torch.Tensor, b: torch.Tensor, dtype):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    err = float(np.max(np.abs(a - b))) if a.size else 0.0
    bound = F32_RTOL * max(float(np.max(np.abs(b))), 1e-30) if dtype == torch.float32 else BF16_ATOL
    assert np.all(np.isfinite(a)) and err <= bound, (err, bound)


# (dtype, head_dim, temporal RoPE pairs, frames of each insert call per segment).  A
# call's frames split into fused passes of at most 4 that never cross an insert, so
# (2, 4) and (5,) make two passes per consolidate; RoPE adds the re-phase kernel.
CASES = [(torch.bfloat16, 128, 0, (3,)), (torch.float32, 64, 0, (3,)),
         (torch.bfloat16, 128, 22, (3,)), (torch.float32, 64, 8, (2, 4)), (torch.bfloat16, 128, 0, (5,))]


@pytest.mark.parametrize("dtype,D,rope,chunks", CASES)
def test_consolidate_noalloc_matches_consolidate(cuda_lib, dtype, D, rope, chunks):
    from paper_2606_10671_gb300 import FadeMem, capi
    lib = capi.load(cuda_lib)
    M, H, N, L = 5, 3, 100, 2
    ref = FadeMem(M, H, D, N, num_layers=L, beta=0.3, dtype=dtype, rope_pairs=rope)
    new = FadeMem(M, H, D, N, num_layers=L, beta=0.3, dtype=dtype, rope_pairs=rope)
    stream = torch.cuda.current_stream()
    sp = ctypes.c_void_p(int(stream.cuda_stream))
    gens = [(HostAR1((N, H, D), 3, KIND_K, l), HostAR1((N, H, D), 3, KIND_V, l)) for l in range(L)]
    per_seg = sum(chunks)
    for seg in range(9):  # 27+ frames through a 5-entry budget: merges in every call from the 2nd on
        keep = []
        for l, (gk, gv) in enumerate(gens):
            K = torch.from_numpy(np.stack([gk.next() for _ in range(per_seg)])).to(dtype).cuda()
            V = torch.from_numpy(np.stack([gv.next() for _ in range(per_seg)])).to(dtype).cuda()
            keep.append((K, V))
            a = 0
            for n in chunks:
                Kc, Vc = K[a:a + n].contiguous(), V[a:a + n].contiguous()
                keep.append((Kc, Vc))
                a += n
                for mem in (ref, new):
                    assert lib.fademem_insert(ctypes.c_void_p(mem.handle), l, ctypes.c_void_p(Kc.data_ptr()),
                                              ctypes.c_void_p(Vc.data_ptr()), n) == capi.FADEMEM_OK
        assert lib.fademem_consolidate(ctypes.c_void_p(ref.handle), sp) == capi.FADEMEM_OK
        st = lib.fademem_consolidate_noalloc(ctypes.c_void_p(new.handle), sp)
        assert st == capi.FADEMEM_OK, capi.fademem_last_error()
        torch.cuda.synchronize()
        for a, b in zip(new.entries(), ref.entries()):
            assert a.tolist() == b.tolist()
        assert new.last_plan() == ref.last_plan()
        count = ref.counts()[0]
        assert new.counts() == ref.counts()
        for l in range(L):
            for x, y in zip(new.layer_memory(l), ref.layer_memory(l)):
                _close(x[:, :count], y[:, :count], dtype)  # occupied slots only
        if seg == 0:
            b0 = new.stats()[1]
        elif seg == 1:
            assert new.stats()[1] - b0 == len(chunks) + (1 if chunks == (5,) else 0)  # passes per call
        Q = torch.from_numpy(host_queries((150, H, D), 3, 0, seg)).to(dtype).cuda()
        for l in range(L):
            _close(new.attend(l, Q), ref.attend(l, Q), dtype)
    assert new.device_status()[1] == 0 and ref.device_status()[1] == 0
