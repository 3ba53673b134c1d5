// Internal declarations of the FadeMem CUDA library (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/fademem.h"

namespace fademem {

// Frames fused into one schedule + consolidation pass.  A pass of F frames
// changes at most 2F slots (merged entry + new entry per frame) and reads at
// most 3F sources (two old blocks per merge + one new frame each).
constexpr int kMaxPassFrames = 4;
constexpr int kMaxDest = 2 * kMaxPassFrames;
constexpr int kMaxSrc = 3 * kMaxPassFrames;
constexpr int kMaxEntries = FADEMEM_MAX_BUDGET + 1;
constexpr int kMaxRopePairs = 64;  // head_dim / 2 at head_dim 128

// Device status word bits (fademem_get_device_status).
constexpr uint32_t kStatusTimeout = FADEMEM_STATUS_TIMEOUT;              // a bounded mbarrier wait gave up
constexpr uint32_t kStatusCountMismatch = FADEMEM_STATUS_COUNT_MISMATCH;  // host and device entry counts disagree
constexpr uint32_t kStatusPlanOverflow = FADEMEM_STATUS_PLAN_OVERFLOW;    // merge plan exceeded its static bounds
// A schedule decision whose best and second-best warped gaps lie within the
// fp64 evaluation error of each other (and are not exact): another correct fp64
// evaluation of u(d) = d^beta could pick the other pair.  The frame of the first
// such decision is kept at byte kNearTieFrameOffset of the workspace (frame + 1).
constexpr uint32_t kStatusNearTie = FADEMEM_STATUS_NEAR_TIE;
constexpr size_t kNearTieFrameOffset = 24;  // after the status word and the two counters

// Device bounds checks.  Built with -DFADEMEM_DEBUG_BOUNDS (build.py
// --debug-bounds, libfademem_debug.so), every kernel checks each global-memory
// access against the buffer it belongs to and each table index against its
// array; an access that fails is skipped and recorded as kStatusBounds in the
// status word.  In the release build kBoundsChecks is false and every check
// compiles away.
#ifdef FADEMEM_DEBUG_BOUNDS
constexpr bool kBoundsChecks = true;
#else
constexpr bool kBoundsChecks = false;
#endif
constexpr uint32_t kStatusBounds = FADEMEM_STATUS_BOUNDS;

// The byte range [lo, hi) of one device buffer.
struct DevRange {
  const char* lo;
  const char* hi;
};
__host__ __device__ inline DevRange dev_range(const void* base, size_t bytes) {
  const char* p = static_cast<const char*>(base);
  return DevRange{p, p + bytes};
}
// True if [p, p + bytes) lies in r (no pointer arithmetic that could wrap).
__host__ __device__ inline bool range_holds(const DevRange& r, const void* p, size_t bytes) {
  const char* c = static_cast<const char*>(p);
  return c >= r.lo && c <= r.hi && (size_t)(r.hi - c) >= bytes;
}
#ifdef __CUDACC__
// True if [p, p + bytes) lies in r; otherwise records kStatusBounds.
__device__ __forceinline__ bool bounds_ok(const DevRange& r, const void* p, size_t bytes, unsigned int* status) {
  if (range_holds(r, p, bytes)) return true;
  atomicOr(status, kStatusBounds);
  return false;
}
// Thread-block cluster helpers (distributed shared memory), for kernels that
// split one tile's keys over a cluster and combine the partials.
// Shared-memory address of the same variable in block `rank` of the cluster.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(r)
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))), "r"(rank));
  return r;
}
__device__ __forceinline__ float ld_cluster(uint32_t a) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ float4 ld_cluster4(uint32_t a) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(a)
               : "memory");
  return v;
}
// Every thread of every block of the cluster arrives (release) and waits
// (acquire): shared-memory writes before it are visible cluster-wide after it.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// True if 0 <= i < n; otherwise records kStatusBounds.
__device__ __forceinline__ bool index_ok(long long i, long long n, unsigned int* status) {
  if (i >= 0 && i < n) return true;
  atomicOr(status, kStatusBounds);
  return false;
}
#endif

// Entry table of the memory (Sec. 3.3 "memory entries"), temporal order.
struct DevMeta {
  int count;
  int pad0;
  long long t_next;                  // index of the next unit (frames seen)
  int slot[kMaxEntries];             // storage slot of entry i
  long long first[kMaxEntries];      // first unit summarised
  long long span[kMaxEntries];       // s
  double mu[kMaxEntries];            // temporal centre
};

// Fused merge plan of one pass.  Destination d receives
//   sum_k w_k * source_k   (linear operators)   or   max_k source_k (max pooling)
// over its sources, which are stored contiguously and in destination order.
// A source is an old slot (ref >= 0, its content before the pass) or a new
// frame of the pass (ref = -(f + 1)).
struct DevPlan {
  int n_src;
  int n_dest;
  int frames;
  int op;
  int src_ref[kMaxSrc];
  float src_w[kMaxSrc];
  int src_dest[kMaxSrc];
  int dest_slot[kMaxDest];
  int merged_pair[kMaxPassFrames];   // j chosen for each frame (-1: no merge)
  long long near_tie_t;              // first frame of the pass decided on a near-tie, -1 if none
};

struct DevState {
  DevMeta meta;
  DevPlan plan;
};

// Layout of one layer in the workspace: K then V, each [H][M][N][D], then
// (temporal RoPE only) the attention keys K_att [H][M][N][D].
struct Geometry {
  int L, H, M, N, D;
  int dtype;             // fademem_dtype
  size_t elem;           // bytes per element
  size_t slab_elems;     // N * D
  size_t kv_elems;       // H * M * N * D (one of K or V of one layer)
  size_t state_bytes;    // status word + two DevState buffers, each rounded to 256
  size_t layer_bytes;    // (2 or 3) * kv_elems * elem, rounded to 256
  size_t total_bytes;
  int rope_pairs;        // temporal RoPE pairs P (0: off)
  double rope_omega[kMaxRopePairs];  // omega_k = theta^(-k/P)
};

// Per-pass source pointers: layer l's K (or V) frames of the pass start at
// src[l][0] (K) / src[l][1] (V), frames contiguous ([F*N][H][D]).
struct PassSources {
  const void* src[FADEMEM_MAX_LAYERS][2];
};

// Schedules one pass of `frames` units: reads in->meta, writes out->meta and
// out->plan (in == out for an in-place pass).  expected_count: the host's
// entry count before the pass (count = min(frames, M)); a mismatch sets
// kStatusCountMismatch in *status and leaves an empty plan.
cudaError_t launch_schedule(const DevState* in, DevState* out, unsigned int* status, int frames, int M, double beta,
                            int anchor, int op, int expected_count, cudaStream_t stream);
// Schedule of the next pass computed inside the consolidation kernel (by one
// extra block) from the entry table `in` into `out`; out == nullptr skips it.
// Temporal RoPE of one consolidation pass: frame f of the pass sits at
// position t0 + f; K frame sources are rotated by -(t0 + f) omega_k as they
// are loaded (stored keys carry no phase).
struct PassRope {
  int pairs;             // 0: no rotation
  long long t0;
  double omega[kMaxRopePairs];
};

struct Lookahead {
  const DevState* in;
  DevState* out;
  unsigned int* status;
  unsigned long long* totals;  // consolidation counters: [blocks moved, passes]
  int frames, expected_count, anchor, op;
  double beta;
};
cudaError_t launch_consolidate(const Geometry& g, void* cache_base, const DevState* st, const PassSources& srcs,
                               int frames, int op, const Lookahead& la, const PassRope& rope, cudaStream_t stream);
// Temporal RoPE re-index: for every layer, head and entry i < count of st's
// entry table, K_att[slot_i] = stored K[slot_i] rotated to position
// t_next - count + i (the rest of each row copied unchanged).
cudaError_t launch_rephase(const Geometry& g, void* cache_base, const DevState* st, int count, long long t_next,
                           unsigned int* status, cudaStream_t stream);
// Attention over Lk memory keys (Kc/Vc: one layer's [H][M][N][D] memory) followed
// by Lk2 current-chunk keys (Kcur/Vcur: [Lk2][H][D]); either count may be 0.
cudaError_t launch_attend_f32(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur,
                              const void* Vcur, int Lk2, const float* Q, float* out, int Lq, float scale,
                              unsigned int* status, cudaStream_t stream);
// Returns cudaErrorNotSupported if the shape is outside the tensor-core path.
cudaError_t launch_attend_bf16(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur,
                               const void* Vcur, int Lk2, const void* Q, void* out, int Lq, float scale,
                               unsigned int* status, cudaStream_t stream, char* err, size_t errlen);

// Multiprocessor count of the current device, looked up once per device
// (PerDevice table, thread-safe); `fallback` if the query fails.
int current_device_sm_count(int fallback);

// Waits on an mbarrier that is never signalled, through the same bounded wait
// the kernels use; sets kStatusTimeout after limit_cycles.
cudaError_t launch_wait_selftest(unsigned int* status, long long limit_cycles, cudaStream_t stream);

}  // namespace fademem
