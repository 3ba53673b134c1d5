// C ABI of the FadeMem library (include/fademem.h): argument checks, workspace
// layout, the pending-insert list and the split of pending frames into fused
// passes.  All arithmetic of the method runs in the kernels.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>
#include <new>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "fademem_internal.h"
#include "per_device.h"

using namespace fademem;

namespace {

thread_local char g_err[512] = "";

// NVTX range around an entry point, visible in Nsight timelines (a no-op
// unless a tool is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

fademem_status fail(fademem_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

fademem_status cuda_fail(cudaError_t e, const char* what) {
  return fail(FADEMEM_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Chunk {
  const char* K;
  const char* V;
  int frames;
};

}  // namespace

struct fademem_ctx {
  fademem_config cfg;
  Geometry g;
  char* ws;
  size_t ws_bytes;
  unsigned int* status;  // device status word (workspace)
  DevState* st_buf[2];   // two entry-table buffers (workspace)
  int cur;               // st_buf[cur] holds the current entry table
  char* cache;
  bool need_init;
  // Schedule lookahead: the consolidation kernel of a single-pass call also
  // schedules the next pass (assuming as many frames) into st_buf[1 - cur].
  bool la_valid;         // st_buf[1 - cur] holds that plan
  int la_frames;         // the frame count it assumed
  bool la_enabled;
  unsigned long long launches = 0;  // kernels this handle launched
  // fademem_step_host: its own compute, host-to-device and device-to-host
  // streams, and per staging slot the events "inputs copied in" (ev_in), "step
  // computed: inputs consumed, output written" (ev_att) and "output copied out"
  // (ev_out); ev_entry marks the caller's stream at entry.
  cudaStream_t comp_stream = nullptr, h2d_stream = nullptr, d2h_stream = nullptr;
  cudaEvent_t ev_entry = nullptr;
  cudaEvent_t ev_in[2] = {nullptr, nullptr};
  cudaEvent_t ev_att[2] = {nullptr, nullptr};
  cudaEvent_t ev_out[2] = {nullptr, nullptr};
  bool slot_used[2] = {false, false};
  int host_slot = 0;
  // The handle's last enqueuing call was fademem_step_host on this stream: the
  // next step needs no wait on the caller's stream (nothing of the handle can
  // have been enqueued there since).  Every other enqueuing entry point clears it.
  bool chained = false;
  cudaStream_t chained_stream = nullptr;
  int count;             // entries, = min(frames, M) (one merge per insert beyond the budget)
  long long frames;      // consolidated frames
  std::vector<Chunk> pending[FADEMEM_MAX_LAYERS];
  int pending_frames[FADEMEM_MAX_LAYERS];
};

static fademem_status check_config(const fademem_config* c, Geometry* g) {
  if (!c) return fail(FADEMEM_ERR_INVALID_ARG, "config is NULL");
  if (c->budget < 2 || c->budget > FADEMEM_MAX_BUDGET)
    return fail(FADEMEM_ERR_INVALID_ARG, "budget must be in [2, %d] (got %d)", FADEMEM_MAX_BUDGET, c->budget);
  if (c->heads < 1 || c->heads > 65535) return fail(FADEMEM_ERR_INVALID_ARG, "heads must be >= 1 (got %d)", c->heads);
  if (c->head_dim != 64 && c->head_dim != 128)
    return fail(FADEMEM_ERR_INVALID_ARG, "head_dim must be 64 or 128 (got %d)", c->head_dim);
  if (c->tokens_per_frame < 1 || c->tokens_per_frame > (1 << 20))
    return fail(FADEMEM_ERR_INVALID_ARG, "tokens_per_frame must be in [1, 2^20] (got %d)", c->tokens_per_frame);
  if (c->num_layers < 1 || c->num_layers > FADEMEM_MAX_LAYERS)
    return fail(FADEMEM_ERR_INVALID_ARG, "num_layers must be in [1, %d] (got %d)", FADEMEM_MAX_LAYERS,
                c->num_layers);
  if (!(c->beta > 0.0 && c->beta <= 1.0)) return fail(FADEMEM_ERR_INVALID_ARG, "beta must be in (0, 1]");
  if (c->anchor != 0 && c->anchor != 1) return fail(FADEMEM_ERR_INVALID_ARG, "anchor must be 0 or 1");
  if (c->merge_op < 0 || c->merge_op > 3) return fail(FADEMEM_ERR_INVALID_ARG, "unknown merge_op %d", c->merge_op);
  if (c->dtype != FADEMEM_F32 && c->dtype != FADEMEM_BF16)
    return fail(FADEMEM_ERR_INVALID_ARG, "unknown dtype %d", c->dtype);
  if (!(c->scale >= 0.f) || isinf(c->scale)) return fail(FADEMEM_ERR_INVALID_ARG, "scale must be finite and >= 0");
  if (c->dtype == FADEMEM_BF16 && c->head_dim != 128)
    return fail(FADEMEM_ERR_UNSUPPORTED, "bf16 storage supports head_dim 128 only");
  const long long lk = (long long)c->budget * c->tokens_per_frame;
  if (lk > (1LL << 30)) return fail(FADEMEM_ERR_INVALID_ARG, "budget * tokens_per_frame too large");
  if ((long long)c->tokens_per_frame * c->heads * c->head_dim >= (1LL << 31))
    return fail(FADEMEM_ERR_INVALID_ARG, "tokens_per_frame * heads * head_dim must be below 2^31");
  if (c->rope_pairs < 0 || 2 * c->rope_pairs > c->head_dim)
    return fail(FADEMEM_ERR_INVALID_ARG, "rope_pairs must be in [0, head_dim / 2] (got %d)", c->rope_pairs);
  if (c->rope_pairs > 0 && !(c->rope_theta == 0.0 || (c->rope_theta > 1.0 && c->rope_theta < 1e30)))
    return fail(FADEMEM_ERR_INVALID_ARG, "rope_theta must be 0 (10000) or above 1");
  if (g) {
    g->L = c->num_layers;
    g->H = c->heads;
    g->M = c->budget;
    g->N = c->tokens_per_frame;
    g->D = c->head_dim;
    g->dtype = c->dtype;
    g->elem = c->dtype == FADEMEM_BF16 ? 2 : 4;
    g->slab_elems = (size_t)g->N * g->D;
    g->kv_elems = (size_t)g->H * g->M * g->slab_elems;
    g->state_bytes = 256 + 2 * round_up(sizeof(DevState), 256);
    g->layer_bytes = round_up((c->rope_pairs > 0 ? 3 : 2) * g->kv_elems * g->elem, 256);
    g->rope_pairs = c->rope_pairs;
    const double theta = c->rope_theta == 0.0 ? 10000.0 : c->rope_theta;
    for (int k = 0; k < kMaxRopePairs; ++k)
      g->rope_omega[k] = k < c->rope_pairs ? pow(theta, -(double)k / (double)c->rope_pairs) : 0.0;
    g->total_bytes = g->state_bytes + (size_t)g->L * g->layer_bytes;
  }
  return FADEMEM_OK;
}

extern "C" {

FADEMEM_API size_t fademem_workspace_bytes(const fademem_config* cfg) {
  Geometry g;
  if (check_config(cfg, &g) != FADEMEM_OK) return 0;
  return g.total_bytes;
}

FADEMEM_API fademem_status fademem_create(const fademem_config* cfg, void* workspace, size_t workspace_bytes,
                                          fademem_t* out) {
  if (!out) return fail(FADEMEM_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  Geometry g;
  fademem_status s = check_config(cfg, &g);
  if (s != FADEMEM_OK) return s;
  if (!workspace) return fail(FADEMEM_ERR_WORKSPACE, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return fail(FADEMEM_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (workspace_bytes < g.total_bytes)
    return fail(FADEMEM_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, g.total_bytes);
  fademem_ctx* h = new (std::nothrow) fademem_ctx();
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "out of host memory");
  h->cfg = *cfg;
  if (h->cfg.scale == 0.f) h->cfg.scale = 1.0f / sqrtf((float)cfg->head_dim);
  if (h->cfg.rope_pairs > 0 && h->cfg.rope_theta == 0.0) h->cfg.rope_theta = 10000.0;  // the documented default
  h->g = g;
  h->ws = reinterpret_cast<char*>(workspace);
  h->ws_bytes = workspace_bytes;
  h->status = reinterpret_cast<unsigned int*>(h->ws);
  h->st_buf[0] = reinterpret_cast<DevState*>(h->ws + 256);
  h->st_buf[1] = reinterpret_cast<DevState*>(h->ws + 256 + round_up(sizeof(DevState), 256));
  h->cur = 0;
  h->cache = h->ws + g.state_bytes;
  h->la_valid = false;
  h->la_frames = 0;
  h->la_enabled = true;
  h->need_init = true;
  h->count = 0;
  h->frames = 0;
  for (int l = 0; l < FADEMEM_MAX_LAYERS; ++l) h->pending_frames[l] = 0;
  *out = h;
  g_err[0] = 0;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_insert(fademem_t h, int layer, const void* K, const void* V, int nframes) {
  NvtxRange nvtx_("fademem_insert");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (layer < 0 || layer >= h->g.L) return fail(FADEMEM_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (!K || !V) return fail(FADEMEM_ERR_INVALID_ARG, "K or V is NULL");
  if (!aligned16(K) || !aligned16(V)) return fail(FADEMEM_ERR_INVALID_ARG, "K and V must be 16-byte aligned");
  if (nframes < 1) return fail(FADEMEM_ERR_INVALID_ARG, "nframes must be >= 1 (got %d)", nframes);
  if (h->pending_frames[layer] + nframes > FADEMEM_MAX_PENDING)
    return fail(FADEMEM_ERR_PENDING, "more than %d frames pending on layer %d", FADEMEM_MAX_PENDING, layer);
  h->pending[layer].push_back(Chunk{reinterpret_cast<const char*>(K), reinterpret_cast<const char*>(V), nframes});
  h->pending_frames[layer] += nframes;
  return FADEMEM_OK;
}

static DevState* cur_state(fademem_t h) { return h->st_buf[h->cur]; }

static fademem_status ensure_init(fademem_t h, cudaStream_t stream) {
  if (!h->need_init) return FADEMEM_OK;
  h->chained = false;
  cudaError_t e = cudaMemsetAsync(h->ws, 0, h->g.state_bytes, stream);
  if (e != cudaSuccess) return cuda_fail(e, "initialising the entry table");
  h->cur = 0;
  h->need_init = false;
  return FADEMEM_OK;
}



FADEMEM_API fademem_status fademem_consolidate(fademem_t h, void* stream_) {
  NvtxRange nvtx_("fademem_consolidate");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  h->chained = false;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  const int L = h->g.L;
  const int F = h->pending_frames[0];
  for (int l = 1; l < L; ++l)
    if (h->pending_frames[l] != F)
      return fail(FADEMEM_ERR_INVALID_ARG, "layer %d has %d pending frames, layer 0 has %d", l,
                  h->pending_frames[l], F);
  if (F == 0) return FADEMEM_OK;
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;

  const size_t frame_bytes = (size_t)h->g.N * h->g.H * h->g.D * h->g.elem;
  // Passes: at most kMaxPassFrames frames each, never crossing an insert boundary.
  std::vector<int> pass_frames;
  {
    std::vector<int> ci(L, 0), co(L, 0);
    int done = 0;
    while (done < F) {
      int nf = F - done < kMaxPassFrames ? F - done : kMaxPassFrames;
      for (int l = 0; l < L; ++l) {
        const int left = h->pending[l][ci[l]].frames - co[l];
        if (left < nf) nf = left;
      }
      pass_frames.push_back(nf);
      for (int l = 0; l < L; ++l) {
        co[l] += nf;
        if (co[l] == h->pending[l][ci[l]].frames) {
          ++ci[l];
          co[l] = 0;
        }
      }
      done += nf;
    }
  }
  // A lookahead schedule fits if it assumed exactly this single pass; it was
  // written by an earlier kernel on this stream, so stream order suffices.
  const bool use_la = h->la_valid && pass_frames.size() == 1 && pass_frames[0] == h->la_frames;
  h->la_valid = false;
  const bool make_la = h->la_enabled && pass_frames.size() == 1;
  std::vector<int> ci(L, 0), co(L, 0);  // chunk index and frame offset inside it, per layer
  PassSources srcs;
  memset(&srcs, 0, sizeof(srcs));
  for (size_t pi = 0; pi < pass_frames.size(); ++pi) {
    const int nf = pass_frames[pi];
    for (int l = 0; l < L; ++l) {
      const Chunk& c = h->pending[l][ci[l]];
      srcs.src[l][0] = c.K + (size_t)co[l] * frame_bytes;
      srcs.src[l][1] = c.V + (size_t)co[l] * frame_bytes;
    }
    cudaError_t e;
    if (pi == 0 && use_la) {
      h->cur ^= 1;  // the lookahead already wrote this pass's entry table and plan
    } else {
      e = launch_schedule(cur_state(h), cur_state(h), h->status, nf, h->g.M, h->cfg.beta, h->cfg.anchor,
                          h->cfg.merge_op, h->count, stream);
      if (e != cudaSuccess) return cuda_fail(e, "launching the schedule kernel");
      ++h->launches;
    }
    const long long frames_after = h->frames + nf;
    const int count_after = frames_after < h->g.M ? (int)frames_after : h->g.M;
    Lookahead la;
    la.in = cur_state(h);
    la.out = make_la ? h->st_buf[h->cur ^ 1] : nullptr;
    la.status = h->status;
    la.totals = reinterpret_cast<unsigned long long*>(h->ws + 8);
    la.frames = nf;
    la.expected_count = count_after;
    la.anchor = h->cfg.anchor;
    la.op = h->cfg.merge_op;
    la.beta = h->cfg.beta;
    PassRope rope;
    rope.pairs = h->g.rope_pairs;
    rope.t0 = h->frames;
    memcpy(rope.omega, h->g.rope_omega, sizeof(rope.omega));
    e = launch_consolidate(h->g, h->cache, cur_state(h), srcs, nf, h->cfg.merge_op, la, rope, stream);
    if (e != cudaSuccess) return cuda_fail(e, "launching the consolidation kernel");
    ++h->launches;
    h->frames = frames_after;
    h->count = count_after;
    for (int l = 0; l < L; ++l) {
      co[l] += nf;
      if (co[l] == h->pending[l][ci[l]].frames) {
        ++ci[l];
        co[l] = 0;
      }
    }
  }
  for (int l = 0; l < L; ++l) {
    h->pending[l].clear();
    h->pending_frames[l] = 0;
  }
  if (h->g.rope_pairs > 0) {
    // Keys for attention: every entry rotated to its re-indexed position.
    cudaError_t e = launch_rephase(h->g, h->cache, cur_state(h), h->count, h->frames, h->status, stream);
    if (e != cudaSuccess) return cuda_fail(e, "launching the re-phase kernel");
    ++h->launches;
  }
  if (make_la) {
    h->la_valid = true;
    h->la_frames = F;
  }
  return FADEMEM_OK;
}

static fademem_status attend_impl(fademem_t h, int layer, const void* Q, const void* Kcur, const void* Vcur,
                                  int ncur, void* out, int Lq, void* stream_) {
  NvtxRange nvtx_(ncur > 0 ? "fademem_attend_ext" : "fademem_attend");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  h->chained = false;
  if (layer < 0 || layer >= h->g.L) return fail(FADEMEM_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (!Q || !out) return fail(FADEMEM_ERR_INVALID_ARG, "Q or out is NULL");
  if (!aligned16(Q) || !aligned16(out)) return fail(FADEMEM_ERR_INVALID_ARG, "Q and out must be 16-byte aligned");
  if (Lq < 1 || Lq > (1 << 24)) return fail(FADEMEM_ERR_INVALID_ARG, "Lq must be in [1, 2^24] (got %d)", Lq);
  if (ncur < 0 || ncur > (1 << 24)) return fail(FADEMEM_ERR_INVALID_ARG, "ncur must be in [0, 2^24] (got %d)", ncur);
  if (ncur > 0 && (!Kcur || !Vcur)) return fail(FADEMEM_ERR_INVALID_ARG, "Kcur or Vcur is NULL");
  if (ncur > 0 && (!aligned16(Kcur) || !aligned16(Vcur)))
    return fail(FADEMEM_ERR_INVALID_ARG, "Kcur and Vcur must be 16-byte aligned");
  for (int l = 0; l < h->g.L; ++l)
    if (h->pending_frames[l] != 0)
      return fail(FADEMEM_ERR_PENDING, "frames inserted on layer %d await fademem_consolidate", l);
  if (h->count == 0 && ncur == 0) return fail(FADEMEM_ERR_EMPTY, "the memory holds no entries");
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  const int Lk = h->count * h->g.N;
  const char* Kmem = h->cache + (size_t)layer * h->g.layer_bytes;
  const char* Vc = Kmem + h->g.kv_elems * h->g.elem;
  // With temporal RoPE, attention reads the re-indexed keys (after V).
  const char* Kc = h->g.rope_pairs > 0 ? Vc + h->g.kv_elems * h->g.elem : Kmem;
  cudaError_t e;
  if (h->g.dtype == FADEMEM_F32) {
    e = launch_attend_f32(h->g, Kc, Vc, Lk, Kcur, Vcur, ncur, reinterpret_cast<const float*>(Q),
                          reinterpret_cast<float*>(out), Lq, h->cfg.scale, h->status, stream);
  } else {
    char msg[256] = "";
    e = launch_attend_bf16(h->g, Kc, Vc, Lk, Kcur, Vcur, ncur, Q, out, Lq, h->cfg.scale, h->status, stream, msg,
                           sizeof(msg));
    if (e == cudaErrorNotSupported) return fail(FADEMEM_ERR_UNSUPPORTED, "%s", msg);
    if (e == cudaErrorInvalidValue && msg[0]) return fail(FADEMEM_ERR_INVALID_ARG, "%s", msg);
  }
  if (e != cudaSuccess) return cuda_fail(e, "launching the attention kernel");
  ++h->launches;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_attend(fademem_t h, int layer, const void* Q, void* out, int Lq, void* stream_) {
  return attend_impl(h, layer, Q, nullptr, nullptr, 0, out, Lq, stream_);
}

FADEMEM_API fademem_status fademem_attend_ext(fademem_t h, int layer, const void* Q, const void* Kcur,
                                              const void* Vcur, int ncur, void* out, int Lq, void* stream_) {
  return attend_impl(h, layer, Q, Kcur, Vcur, ncur, out, Lq, stream_);
}

FADEMEM_API fademem_status fademem_counts(fademem_t h, int* count, int64_t* frames_seen) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (count) *count = h->count;
  if (frames_seen) *frames_seen = h->frames;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_get_entries(fademem_t h, void* stream_, int capacity, int* count, int32_t* slot,
                                               int64_t* first, int64_t* span, int64_t* mu2) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (!count) return fail(FADEMEM_ERR_INVALID_ARG, "count is NULL");
  if (capacity < h->count) return fail(FADEMEM_ERR_INVALID_ARG, "capacity %d < %d entries", capacity, h->count);
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  DevMeta m;
  e = cudaMemcpy(&m, &cur_state(h)->meta, sizeof(m), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the entry table");
  if (m.count < 0 || m.count > kMaxEntries)
    return fail(FADEMEM_ERR_DEVICE_CHECK, "device entry count %d is out of range", m.count);
  if (m.count > capacity) return fail(FADEMEM_ERR_INVALID_ARG, "capacity %d < %d entries", capacity, m.count);
  *count = m.count;
  for (int i = 0; i < m.count; ++i) {
    if (slot) slot[i] = m.slot[i];
    if (first) first[i] = m.first[i];
    if (span) span[i] = m.span[i];
    if (mu2) mu2[i] = (int64_t)llround(2.0 * m.mu[i]);
  }
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_last_plan(fademem_t h, void* stream_, int* n_src, int* n_dest, int* frames) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  DevPlan p;
  e = cudaMemcpy(&p, &cur_state(h)->plan, sizeof(p), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the merge plan");
  if (n_src) *n_src = p.n_src;
  if (n_dest) *n_dest = p.n_dest;
  if (frames) *frames = p.frames;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_stats(fademem_t h, void* stream_, uint64_t* blocks_moved, uint64_t* passes,
                                        uint64_t* kernel_launches) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  unsigned long long t[2] = {0, 0};
  e = cudaMemcpy(t, h->ws + 8, sizeof(t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the consolidation counters");
  if (blocks_moved) *blocks_moved = t[0];
  if (passes) *passes = t[1];
  if (kernel_launches) *kernel_launches = h->launches;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_layer_memory(fademem_t h, int layer, void** K, void** V) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (layer < 0 || layer >= h->g.L) return fail(FADEMEM_ERR_INVALID_ARG, "layer %d out of range", layer);
  char* k = h->cache + (size_t)layer * h->g.layer_bytes;
  if (K) *K = k;
  if (V) *V = k + h->g.kv_elems * h->g.elem;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_get_device_status(fademem_t h, void* stream_, uint32_t* word) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  unsigned int w = 0;
  e = cudaMemcpy(&w, h->status, sizeof(w), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the device status");
  unsigned long long tie = 0;  // frame + 1 of the first uncertified schedule decision
  char* tie_slot = reinterpret_cast<char*>(h->status) + kNearTieFrameOffset;
  if (w & kStatusNearTie) {
    e = cudaMemcpy(&tie, tie_slot, sizeof(tie), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device status");
  }
  const unsigned int zero = 0;
  e = cudaMemcpy(h->status, &zero, sizeof(zero), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "clearing the device status");
  const unsigned long long zero64 = 0;
  e = cudaMemcpy(tie_slot, &zero64, sizeof(zero64), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "clearing the device status");
  if (word) *word = w;
  if (w & kStatusTimeout) return fail(FADEMEM_ERR_DEVICE_TIMEOUT, "a device wait timed out (status 0x%x)", w);
  if (w & kStatusNearTie)
    return fail(FADEMEM_ERR_DEVICE_CHECK,
                "%sschedule decision at frame %lld not certified: its two smallest warped gaps are equal within "
                "the fp64 evaluation error of d^beta (status 0x%x)",
                w != kStatusNearTie ? "a device check failed; " : "", (long long)tie - 1, w);
  if (w) return fail(FADEMEM_ERR_DEVICE_CHECK, "a device check failed (status 0x%x)", w);
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_selftest_wait_timeout(fademem_t h, void* stream_) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  h->chained = false;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = launch_wait_selftest(h->status, 2000000LL, stream);  // about 1 ms
  if (e != cudaSuccess) return cuda_fail(e, "launching the wait self-test");
  ++h->launches;
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_reset(fademem_t h, void* stream_) {
  NvtxRange nvtx_("fademem_reset");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  h->chained = false;
  h->la_valid = false;
  h->need_init = true;
  fademem_status s = ensure_init(h, reinterpret_cast<cudaStream_t>(stream_));
  if (s != FADEMEM_OK) return s;
  h->count = 0;
  h->frames = 0;
  for (int l = 0; l < h->g.L; ++l) {
    h->pending[l].clear();
    h->pending_frames[l] = 0;
  }
  return FADEMEM_OK;
}

}  // extern "C"

// ---- Consolidation with library-owned scratch (fademem_consolidate_noalloc) ----
namespace {

// Working copy of one handle's DevState (entry table, merge plan, status word)
// for fademem_consolidate_noalloc.  Host code must not pass this name to a
// kernel: on the host it is only a stand-in; its device address comes from
// cudaGetSymbolAddress, once per device.
static __device__ __align__(256) unsigned char g_noalloc_scratch[FADEMEM_NOALLOC_SCRATCH_BYTES];
// DevState holds the entry table of the largest budget fademem_create accepts
// (kMaxEntries = FADEMEM_MAX_BUDGET + 1), so every handle's state fits.
static_assert(sizeof(DevState) <= FADEMEM_NOALLOC_SCRATCH_BYTES, "DevState must fit the no-alloc scratch");
static_assert(kMaxEntries == FADEMEM_MAX_BUDGET + 1, "the entry table must hold every budget fademem_create accepts");

PerDevice<void*> g_scratch_addr;

fademem_status noalloc_scratch(DevState** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  cudaError_t lookup = cudaSuccess;
  void* p = nullptr;
  const bool ok = g_scratch_addr.get(dev, [&lookup](int, void** v) {
    lookup = cudaGetSymbolAddress(v, g_noalloc_scratch);  // with this device current
    return lookup == cudaSuccess;
  }, &p);
  if (!ok && lookup != cudaSuccess) return cuda_fail(lookup, "looking up the no-alloc scratch");
  if (!ok) return fail(FADEMEM_ERR_UNSUPPORTED, "device %d out of range", dev);
  *out = reinterpret_cast<DevState*>(p);
  return FADEMEM_OK;
}

}  // namespace

extern "C" {

FADEMEM_API fademem_status fademem_consolidate_noalloc(fademem_t h, void* stream_) {
  NvtxRange nvtx_("fademem_consolidate_noalloc");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  h->chained = false;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DevState* scratch = nullptr;
  fademem_status s = noalloc_scratch(&scratch);
  if (s != FADEMEM_OK) return s;
  s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  // A lookahead schedule lives in the workspace's second entry-table buffer:
  // drop it, and schedule in place on the scratch copy instead.
  h->la_valid = false;
  DevState* own = cur_state(h);
  cudaError_t e = cudaMemcpyAsync(scratch, own, sizeof(DevState), cudaMemcpyDeviceToDevice, stream);
  if (e != cudaSuccess) return cuda_fail(e, "copying the entry table to the no-alloc scratch");
  // Run the ordinary consolidation on the scratch copy, then copy the result back.
  h->st_buf[h->cur] = scratch;
  h->la_enabled = false;
  const fademem_status rs = fademem_consolidate(h, stream_);
  h->la_enabled = true;
  h->st_buf[h->cur] = own;
  e = cudaMemcpyAsync(own, scratch, sizeof(DevState), cudaMemcpyDeviceToDevice, stream);
  if (rs != FADEMEM_OK) return rs;
  if (e != cudaSuccess) return cuda_fail(e, "copying the entry table back from the no-alloc scratch");
  return FADEMEM_OK;
}

// Staging layout of fademem_step_host: slot s (s = 0, 1) holds, 256-byte
// aligned, K then V of every layer, then Q, then the output block.
struct HostStaging {
  size_t frame_bytes, q_bytes, slot_bytes, total;
};
static bool host_staging(const Geometry& g, int nframes, int Lq, HostStaging* st) {
  if (nframes < 1 || nframes > FADEMEM_MAX_PENDING || Lq < 1 || Lq > (1 << 24)) return false;
  st->frame_bytes = round_up((size_t)nframes * g.N * g.H * g.D * g.elem, 256);
  st->q_bytes = round_up((size_t)Lq * g.H * g.D * g.elem, 256);
  st->slot_bytes = 2 * (size_t)g.L * st->frame_bytes + 2 * st->q_bytes;
  st->total = 2 * st->slot_bytes;
  return true;
}

FADEMEM_API size_t fademem_host_staging_bytes(const fademem_config* cfg, int nframes, int Lq) {
  Geometry g;
  HostStaging st;
  if (check_config(cfg, &g) != FADEMEM_OK || !host_staging(g, nframes, Lq, &st)) return 0;
  return st.total;
}

FADEMEM_API fademem_status fademem_step_host(fademem_t h, const void* const* K_host, const void* const* V_host,
                                            int nframes, int layer, const void* Q_host, void* out_host, int Lq,
                                            void* staging, size_t staging_bytes, void* stream_) {
  NvtxRange nvtx_("fademem_step_host");
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (!K_host || !V_host || !Q_host || !out_host) return fail(FADEMEM_ERR_INVALID_ARG, "a host pointer is NULL");
  for (int l = 0; l < h->g.L; ++l)
    if (!K_host[l] || !V_host[l]) return fail(FADEMEM_ERR_INVALID_ARG, "K_host[%d] or V_host[%d] is NULL", l, l);
  if (layer < 0 || layer >= h->g.L) return fail(FADEMEM_ERR_INVALID_ARG, "layer %d out of range", layer);
  HostStaging st;
  if (!host_staging(h->g, nframes, Lq, &st))
    return fail(FADEMEM_ERR_INVALID_ARG, "nframes must be in [1, %d] and Lq in [1, 2^24]", FADEMEM_MAX_PENDING);
  if (!staging || !aligned16(staging) || staging_bytes < st.total)
    return fail(FADEMEM_ERR_WORKSPACE, "staging needs %zu bytes, 16-byte aligned (got %zu at %p)", st.total,
                staging_bytes, staging);
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t e;
  if (!h->comp_stream) {
    cudaStream_t* ss[3] = {&h->comp_stream, &h->h2d_stream, &h->d2h_stream};
    for (cudaStream_t* x : ss)
      if ((e = cudaStreamCreateWithFlags(x, cudaStreamNonBlocking)) != cudaSuccess)
        return cuda_fail(e, "creating the step streams");
    if ((e = cudaEventCreateWithFlags(&h->ev_entry, cudaEventDisableTiming)) != cudaSuccess)
      return cuda_fail(e, "creating the step events");
    for (int k = 0; k < 2; ++k)
      if ((e = cudaEventCreateWithFlags(&h->ev_in[k], cudaEventDisableTiming)) != cudaSuccess ||
          (e = cudaEventCreateWithFlags(&h->ev_att[k], cudaEventDisableTiming)) != cudaSuccess ||
          (e = cudaEventCreateWithFlags(&h->ev_out[k], cudaEventDisableTiming)) != cudaSuccess)
        return cuda_fail(e, "creating the step events");
  }
  const int s = h->host_slot;
  char* slot = static_cast<char*>(staging) + s * st.slot_bytes;
  char* dq = slot + 2 * (size_t)h->g.L * st.frame_bytes;
  char* dout = dq + st.q_bytes;
  const size_t fb = (size_t)nframes * h->g.N * h->g.H * h->g.D * h->g.elem;
  const size_t qb = (size_t)Lq * h->g.H * h->g.D * h->g.elem;
  // The step follows what was enqueued on `stream` before it, unless the
  // previous call was a step on the same stream (then `stream` only waits for
  // that step's output, and waiting on it would serialise consecutive steps).
  if (!(h->chained && h->chained_stream == stream)) {
    if ((e = cudaEventRecord(h->ev_entry, stream)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(h->h2d_stream, h->ev_entry, 0)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(h->comp_stream, h->ev_entry, 0)) != cudaSuccess)
      return cuda_fail(e, "ordering the step streams");
  }
  // Inputs into slot s, once the step before last has consumed them.
  if (h->slot_used[s] && (e = cudaStreamWaitEvent(h->h2d_stream, h->ev_att[s], 0)) != cudaSuccess)
    return cuda_fail(e, "ordering the copy stream");
  for (int l = 0; l < h->g.L; ++l) {
    char* dk = slot + (size_t)(2 * l) * st.frame_bytes;
    if ((e = cudaMemcpyAsync(dk, K_host[l], fb, cudaMemcpyHostToDevice, h->h2d_stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dk + st.frame_bytes, V_host[l], fb, cudaMemcpyHostToDevice, h->h2d_stream)) !=
            cudaSuccess)
      return cuda_fail(e, "copying K/V to the device");
  }
  if ((e = cudaMemcpyAsync(dq, Q_host, qb, cudaMemcpyHostToDevice, h->h2d_stream)) != cudaSuccess)
    return cuda_fail(e, "copying Q to the device");
  if ((e = cudaEventRecord(h->ev_in[s], h->h2d_stream)) != cudaSuccess ||
      (e = cudaStreamWaitEvent(h->comp_stream, h->ev_in[s], 0)) != cudaSuccess)
    return cuda_fail(e, "ordering the compute stream");
  // The output block of slot s is free once the step before last has copied it out.
  if (h->slot_used[s] && (e = cudaStreamWaitEvent(h->comp_stream, h->ev_out[s], 0)) != cudaSuccess)
    return cuda_fail(e, "ordering the compute stream");
  void* cs = reinterpret_cast<void*>(h->comp_stream);
  fademem_status r;
  for (int l = 0; l < h->g.L; ++l) {
    char* dk = slot + (size_t)(2 * l) * st.frame_bytes;
    if ((r = fademem_insert(h, l, dk, dk + st.frame_bytes, nframes)) != FADEMEM_OK) return r;
  }
  if ((r = fademem_consolidate(h, cs)) != FADEMEM_OK) return r;
  if ((r = fademem_attend(h, layer, dq, dout, Lq, cs)) != FADEMEM_OK) return r;
  if ((e = cudaEventRecord(h->ev_att[s], h->comp_stream)) != cudaSuccess ||
      (e = cudaStreamWaitEvent(h->d2h_stream, h->ev_att[s], 0)) != cudaSuccess)
    return cuda_fail(e, "ordering the output copy");
  if ((e = cudaMemcpyAsync(out_host, dout, qb, cudaMemcpyDeviceToHost, h->d2h_stream)) != cudaSuccess)
    return cuda_fail(e, "copying the output to the host");
  // The caller's stream continues once the output is on the host; the next
  // step's kernels do not wait for this copy (they use the other slot).
  if ((e = cudaEventRecord(h->ev_out[s], h->d2h_stream)) != cudaSuccess ||
      (e = cudaStreamWaitEvent(stream, h->ev_out[s], 0)) != cudaSuccess)
    return cuda_fail(e, "ordering the caller's stream");
  h->slot_used[s] = true;
  h->host_slot = s ^ 1;
  h->chained = true;
  h->chained_stream = stream;
  return FADEMEM_OK;
}

// Snapshot layout: SnapshotHeader, then the entry table (DevMeta), then for
// every layer its stored K and V blocks ([H][M][N][D] each), all packed.
struct SnapshotHeader {
  char magic[8];            // "FADEMEM" + '\0'
  uint32_t version;         // 1
  uint32_t header_bytes;    // sizeof(SnapshotHeader)
  fademem_config cfg;
  int32_t count;
  int32_t pad;
  int64_t frames;
  uint64_t meta_bytes;      // sizeof(DevMeta)
  uint64_t kv_bytes;        // bytes of one layer's K (or V) block
};
static const char kSnapshotMagic[8] = {'F', 'A', 'D', 'E', 'M', 'E', 'M', 0};

static bool same_config(const fademem_config& a, const fademem_config& b) {
  return a.budget == b.budget && a.heads == b.heads && a.head_dim == b.head_dim &&
         a.tokens_per_frame == b.tokens_per_frame && a.num_layers == b.num_layers && a.beta == b.beta &&
         a.anchor == b.anchor && a.merge_op == b.merge_op && a.dtype == b.dtype && a.scale == b.scale &&
         a.rope_pairs == b.rope_pairs && (a.rope_pairs == 0 || a.rope_theta == b.rope_theta);
}

FADEMEM_API size_t fademem_state_bytes(fademem_t h) {
  if (!h) return 0;
  return sizeof(SnapshotHeader) + sizeof(DevMeta) + 2 * (size_t)h->g.L * h->g.kv_elems * h->g.elem;
}

FADEMEM_API fademem_status fademem_export_state(fademem_t h, void* host_buf, size_t bytes, void* stream_) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (!host_buf) return fail(FADEMEM_ERR_INVALID_ARG, "host buffer is NULL");
  if (bytes < fademem_state_bytes(h))
    return fail(FADEMEM_ERR_WORKSPACE, "snapshot needs %zu bytes (got %zu)", fademem_state_bytes(h), bytes);
  for (int l = 0; l < h->g.L; ++l)
    if (h->pending_frames[l] != 0)
      return fail(FADEMEM_ERR_PENDING, "frames inserted on layer %d await fademem_consolidate", l);
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  fademem_status s = ensure_init(h, stream);
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  char* out = static_cast<char*>(host_buf);
  SnapshotHeader hd;
  memset(&hd, 0, sizeof(hd));
  memcpy(hd.magic, kSnapshotMagic, sizeof(hd.magic));
  hd.version = 1;
  hd.header_bytes = sizeof(SnapshotHeader);
  hd.cfg = h->cfg;
  hd.count = h->count;
  hd.frames = h->frames;
  hd.meta_bytes = sizeof(DevMeta);
  hd.kv_bytes = h->g.kv_elems * h->g.elem;
  memcpy(out, &hd, sizeof(hd));
  out += sizeof(hd);
  if ((e = cudaMemcpy(out, &cur_state(h)->meta, sizeof(DevMeta), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "reading the entry table");
  out += sizeof(DevMeta);
  for (int l = 0; l < h->g.L; ++l) {
    const char* Kl = h->cache + (size_t)l * h->g.layer_bytes;
    if ((e = cudaMemcpy(out, Kl, 2 * hd.kv_bytes, cudaMemcpyDeviceToHost)) != cudaSuccess)
      return cuda_fail(e, "reading the memory");
    out += 2 * hd.kv_bytes;
  }
  return FADEMEM_OK;
}

FADEMEM_API fademem_status fademem_import_state(fademem_t h, const void* host_buf, size_t bytes, void* stream_) {
  if (!h) return fail(FADEMEM_ERR_INVALID_ARG, "handle is NULL");
  if (!host_buf) return fail(FADEMEM_ERR_INVALID_ARG, "host buffer is NULL");
  if (bytes < sizeof(SnapshotHeader)) return fail(FADEMEM_ERR_INVALID_ARG, "not a FadeMem snapshot (too short)");
  SnapshotHeader hd;
  memcpy(&hd, host_buf, sizeof(hd));
  if (memcmp(hd.magic, kSnapshotMagic, sizeof(hd.magic)) != 0)
    return fail(FADEMEM_ERR_INVALID_ARG, "not a FadeMem snapshot (bad magic)");
  if (hd.version != 1 || hd.header_bytes != sizeof(SnapshotHeader) || hd.meta_bytes != sizeof(DevMeta))
    return fail(FADEMEM_ERR_INVALID_ARG, "snapshot of another library version (%u)", hd.version);
  if (!same_config(hd.cfg, h->cfg)) return fail(FADEMEM_ERR_INVALID_ARG, "snapshot of another configuration");
  if (hd.kv_bytes != h->g.kv_elems * h->g.elem || bytes < fademem_state_bytes(h))
    return fail(FADEMEM_ERR_INVALID_ARG, "snapshot size does not match the configuration");
  const char* in = static_cast<const char*>(host_buf) + sizeof(hd);
  DevMeta meta;
  memcpy(&meta, in, sizeof(meta));
  in += sizeof(meta);
  const long long expect = hd.frames < h->g.M ? hd.frames : h->g.M;
  if (hd.frames < 0 || hd.count != expect || meta.count != hd.count || meta.t_next != hd.frames)
    return fail(FADEMEM_ERR_INVALID_ARG, "snapshot entry table is inconsistent (count %d, frames %lld)", hd.count,
                (long long)hd.frames);
  for (int i = 0; i < meta.count; ++i)
    if (meta.slot[i] < 0 || meta.slot[i] >= h->g.M)
      return fail(FADEMEM_ERR_INVALID_ARG, "snapshot entry %d has slot %d", i, meta.slot[i]);
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  h->chained = false;
  h->need_init = true;
  fademem_status s = ensure_init(h, stream);  // clears the status word, counters and both entry tables
  if (s != FADEMEM_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
  if ((e = cudaMemcpy(&cur_state(h)->meta, &meta, sizeof(meta), cudaMemcpyHostToDevice)) != cudaSuccess)
    return cuda_fail(e, "writing the entry table");
  for (int l = 0; l < h->g.L; ++l) {
    char* Kl = h->cache + (size_t)l * h->g.layer_bytes;
    if ((e = cudaMemcpy(Kl, in, 2 * hd.kv_bytes, cudaMemcpyHostToDevice)) != cudaSuccess)
      return cuda_fail(e, "writing the memory");
    in += 2 * hd.kv_bytes;
  }
  for (int l = 0; l < h->g.L; ++l) {
    h->pending[l].clear();
    h->pending_frames[l] = 0;
  }
  h->count = hd.count;
  h->frames = hd.frames;
  h->la_valid = false;
  if (h->g.rope_pairs > 0 && h->count > 0) {
    e = launch_rephase(h->g, h->cache, cur_state(h), h->count, h->frames, h->status, stream);
    if (e != cudaSuccess) return cuda_fail(e, "launching the re-phase kernel");
    ++h->launches;
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "rebuilding the attention keys");
  }
  return FADEMEM_OK;
}

FADEMEM_API void fademem_destroy(fademem_t h) {
  if (!h) return;
  cudaStream_t ss[3] = {h->comp_stream, h->h2d_stream, h->d2h_stream};
  for (cudaStream_t x : ss) {
    if (x) {
      cudaStreamSynchronize(x);
      cudaStreamDestroy(x);
    }
  }
  if (h->ev_entry) cudaEventDestroy(h->ev_entry);
  for (int s = 0; s < 2; ++s) {
    if (h->ev_in[s]) cudaEventDestroy(h->ev_in[s]);
    if (h->ev_att[s]) cudaEventDestroy(h->ev_att[s]);
    if (h->ev_out[s]) cudaEventDestroy(h->ev_out[s]);
  }
  delete h;
}

FADEMEM_API const char* fademem_last_error(void) { return g_err; }

FADEMEM_API uint32_t fademem_build_flags(void) { return kBoundsChecks ? FADEMEM_BUILD_DEBUG_BOUNDS : 0u; }

}  // extern "C"
