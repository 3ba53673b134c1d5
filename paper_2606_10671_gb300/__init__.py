"""GB300-native FadeMem memory step (arxiv 2606.10671): Python binding of libfademem.so.

``FadeMem`` allocates the device workspace with PyTorch and forwards every call
to the C ABI (``capi``); the schedule, consolidation and attention all run in
the library's CUDA kernels.  Importing works without a GPU; any call that
needs the library fails loudly if it has not been built.
"""
from __future__ import annotations

import torch

from . import capi

_DTYPES = {torch.float32: capi.FADEMEM_F32, torch.bfloat16: capi.FADEMEM_BF16}
_OPS = {"weighted": capi.FADEMEM_MERGE_WEIGHTED, "average": capi.FADEMEM_MERGE_AVERAGE,
        "select_nearest": capi.FADEMEM_MERGE_SELECT_NEAREST, "max_pool": capi.FADEMEM_MERGE_MAX_POOL}


def make_config(budget, heads, head_dim, tokens_per_frame, num_layers=1, beta=0.3, anchor=True, merge_op="weighted",
                dtype=torch.bfloat16, scale=0.0, rope_pairs=0, rope_theta=0.0) -> capi.fademem_config:
    return capi.fademem_config(budget=int(budget), heads=int(heads), head_dim=int(head_dim),
                               tokens_per_frame=int(tokens_per_frame), num_layers=int(num_layers), beta=float(beta),
                               anchor=int(bool(anchor)), merge_op=_OPS[merge_op], dtype=_DTYPES[dtype],
                               scale=float(scale), rope_pairs=int(rope_pairs), rope_theta=float(rope_theta))


def _stream_handle(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


class FadeMem:
    """One FadeMem memory over ``num_layers`` layers (Sec. 3.1), on one CUDA device.

    insert(layer, K, V) registers K/V frames [F*N, H, D] (or [F, N, H, D]);
    consolidate() runs Algorithm S1 for every pending frame on the device;
    attend(layer, Q) returns softmax(scale Q K^T) V over the memory, Q [Lq, H, D].
    """

    def __init__(self, budget, heads, head_dim, tokens_per_frame, num_layers=1, beta=0.3, anchor=True,
                 merge_op="weighted", dtype=torch.bfloat16, scale=0.0, device="cuda", rope_pairs=0, rope_theta=0.0):
        self.cfg = make_config(budget, heads, head_dim, tokens_per_frame, num_layers, beta, anchor, merge_op, dtype,
                               scale, rope_pairs, rope_theta)
        self.dtype = dtype
        self.device = torch.device(device)
        nbytes = capi.fademem_workspace_bytes(self.cfg)
        if nbytes == 0:  # invalid configuration: let the library say why
            import ctypes
            h = ctypes.c_void_p()
            capi.check(capi.load().fademem_create(ctypes.byref(self.cfg), None, 0, ctypes.byref(h)))
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.handle = capi.fademem_create(self.cfg, self.workspace.data_ptr(), nbytes)
        self._borrowed = []

    @property
    def budget(self):
        return self.cfg.budget

    def close(self):
        if getattr(self, "handle", None):
            capi.fademem_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check_frames(self, X):
        c = self.cfg
        if X.dtype != self.dtype or X.device.type != "cuda" or not X.is_contiguous():
            raise ValueError("K/V must be contiguous CUDA tensors of the memory's dtype")
        per = c.tokens_per_frame * c.heads * c.head_dim
        if X.numel() % per != 0 or X.numel() == 0:
            raise ValueError(f"K/V must hold whole frames of {c.tokens_per_frame}x{c.heads}x{c.head_dim}")
        return X.numel() // per

    def insert(self, layer: int, K: torch.Tensor, V: torch.Tensor):
        f = self._check_frames(K)
        if self._check_frames(V) != f:
            raise ValueError("K and V hold different numbers of frames")
        capi.fademem_insert(self.handle, layer, K.data_ptr(), V.data_ptr(), f)
        self._borrowed += [K, V]  # kept alive until consolidate is enqueued

    def consolidate(self, stream=None):
        capi.fademem_consolidate(self.handle, _stream_handle(stream))
        self._borrowed = []

    def attend(self, layer: int, Q: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        c = self.cfg
        if Q.dtype != self.dtype or Q.device.type != "cuda" or not Q.is_contiguous():
            raise ValueError("Q must be a contiguous CUDA tensor of the memory's dtype")
        per = c.heads * c.head_dim
        if Q.numel() % per != 0 or Q.numel() == 0:
            raise ValueError(f"Q must be [Lq, {c.heads}, {c.head_dim}]")
        Lq = Q.numel() // per
        if out is None:
            out = torch.empty((Lq, c.heads, c.head_dim), dtype=self.dtype, device=Q.device)
        capi.fademem_attend(self.handle, layer, Q.data_ptr(), out.data_ptr(), Lq, _stream_handle(stream))
        return out

    def attend_ext(self, layer: int, Q: torch.Tensor, Kcur: torch.Tensor, Vcur: torch.Tensor,
                   out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """Attention over the memory followed by the current chunk's tokens Kcur/Vcur [ncur, H, D]."""
        c = self.cfg
        per = c.heads * c.head_dim
        for X in (Q, Kcur, Vcur):
            if X.dtype != self.dtype or X.device.type != "cuda" or not X.is_contiguous() or X.numel() % per:
                raise ValueError("Q, Kcur and Vcur must be contiguous CUDA tensors [tokens, H, D] of the memory's dtype")
        if Kcur.numel() != Vcur.numel():
            raise ValueError("Kcur and Vcur hold different numbers of tokens")
        Lq, ncur = Q.numel() // per, Kcur.numel() // per
        if out is None:
            out = torch.empty((Lq, c.heads, c.head_dim), dtype=self.dtype, device=Q.device)
        capi.fademem_attend_ext(self.handle, layer, Q.data_ptr(), Kcur.data_ptr(), Vcur.data_ptr(), ncur,
                                out.data_ptr(), Lq, _stream_handle(stream))
        return out

    def step_host(self, Ks, Vs, Q: torch.Tensor, out: torch.Tensor, layer: int = 0, stream=None) -> torch.Tensor:
        """One serving step with host tensors: Ks[l], Vs[l] [nframes*N, H, D] per layer and Q [Lq, H, D]
        (CPU, preferably pinned) in, out [Lq, H, D] (CPU) written once `stream` has synchronised.
        Copies, insert, consolidate and attend all run inside the library (fademem_step_host)."""
        c = self.cfg
        if len(Ks) != c.num_layers or len(Vs) != c.num_layers:
            raise ValueError(f"need K and V for each of the {c.num_layers} layers")
        per_frame = c.tokens_per_frame * c.heads * c.head_dim
        for X in list(Ks) + list(Vs) + [Q, out]:
            if X.device.type != "cpu" or X.dtype != self.dtype or not X.is_contiguous():
                raise ValueError("step_host takes contiguous CPU tensors of the memory's dtype")
        nframes = Ks[0].numel() // per_frame
        if any(X.numel() != nframes * per_frame for X in list(Ks) + list(Vs)) or nframes == 0:
            raise ValueError("every K and V must hold the same whole number of frames")
        Lq = Q.numel() // (c.heads * c.head_dim)
        if Q.numel() != Lq * c.heads * c.head_dim or out.numel() != Q.numel():
            raise ValueError(f"Q and out must be [Lq, {c.heads}, {c.head_dim}]")
        nbytes = capi.fademem_host_staging_bytes(self.cfg, nframes, Lq)
        st = getattr(self, "_staging", None)
        if st is None or st.numel() < nbytes:
            torch.cuda.synchronize(self.device)  # the old staging may still be in use
            self._staging = st = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        capi.fademem_step_host(self.handle, [K.data_ptr() for K in Ks], [V.data_ptr() for V in Vs], nframes, layer,
                               Q.data_ptr(), out.data_ptr(), Lq, st.data_ptr(), st.numel(), _stream_handle(stream))
        return out

    def counts(self):
        return capi.fademem_counts(self.handle)

    def entries(self, stream=None):
        """(slot, first, span, mu2) numpy arrays of the device entry table, temporal order."""
        return capi.fademem_get_entries(self.handle, _stream_handle(stream))

    def last_plan(self, stream=None):
        """(n_src, n_dest, frames) of the latest consolidation pass."""
        return capi.fademem_last_plan(self.handle, _stream_handle(stream))

    def stats(self, stream=None):
        """(blocks moved, consolidation passes) since create/reset, kernels launched since create."""
        return capi.fademem_stats(self.handle, _stream_handle(stream))

    def layer_memory(self, layer: int):
        """(K, V) torch views [H, M, N, D] of one layer's stored memory (slots 0..count-1 valid)."""
        c = self.cfg
        kp, vp = capi.fademem_layer_memory(self.handle, layer)
        base = self.workspace.data_ptr()
        esz = torch.empty((), dtype=self.dtype).element_size()
        n = c.heads * c.budget * c.tokens_per_frame * c.head_dim
        flat = self.workspace
        K = flat[kp - base: kp - base + n * esz].view(self.dtype).view(c.heads, c.budget, c.tokens_per_frame,
                                                                        c.head_dim)
        V = flat[vp - base: vp - base + n * esz].view(self.dtype).view(c.heads, c.budget, c.tokens_per_frame,
                                                                        c.head_dim)
        return K, V

    def device_status(self, stream=None, raise_on_error=True):
        return capi.fademem_get_device_status(self.handle, _stream_handle(stream), raise_on_error)

    def export_state(self, stream=None):
        """Snapshot of the memory (entry table and stored K/V of every layer) as host bytes."""
        return capi.fademem_export_state(self.handle, _stream_handle(stream))

    def import_state(self, snapshot, stream=None):
        """Replace the memory with a snapshot from a memory of the same configuration."""
        capi.fademem_import_state(self.handle, snapshot, _stream_handle(stream))

    def reset(self, stream=None):
        capi.fademem_reset(self.handle, _stream_handle(stream))


__all__ = ["FadeMem", "make_config", "capi"]
