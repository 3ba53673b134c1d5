// Schedule (K1) and fused insert + consolidation (K2) of FadeMem's memory
// update (Algorithm S1; Sec. 3.3 "distance-aware scheduling" and
// "consolidation operator").
//
// K1 runs Algorithm S1's bookkeeping for the frames of one pass on the device
// (one warp): append, warped gaps g_i = |(t-mu_{i+1})^beta - (t-mu_i)^beta|
// over the eligible pairs, argmin with the lowest index on ties, span and
// centre update with the first-frame anchor rule, slot compaction.  While
// doing so it tracks, for every entry, which source blocks (old slot contents
// or new frames) its block is made of and with which weight, so the pass
// becomes a plan "slot <- sum_k w_k source_k" (max_k for max pooling).
//
// K2 applies the plan to every layer, K and V, in one pass over HBM: each
// thread owns one 16-byte vector coordinate (layer, K|V, head, token, dims)
// and reads every source of the plan at that coordinate before writing any
// destination, so slots that are both read and rewritten need no second
// buffer.  Each source block is read once and each changed slot written once.
#include <cuda_bf16.h>
#include <math.h>

#include "fademem_internal.h"
#include "per_device.h"

namespace fademem {
namespace {

__device__ __forceinline__ double warp_u(double d, double beta) {
  // u(d) = d^beta.  beta = 1 and beta = 0.5 use the exact forms of the same
  // function (identity, correctly rounded square root), so that exact ties
  // between gaps stay exact ties.
  if (beta == 1.0) return d;
  if (beta == 0.5) return sqrt(d);
  return pow(d, beta);
}

// fp32 estimate of u(d) and a bound on its error.  powf is accurate to a few
// ulp and beta rounded to fp32 moves d^beta by under beta * 2^-24 * ln(d)
// relative, so 2^-16 relative (about 100x the worst case) is a safe bound.
__device__ __forceinline__ float warp_u32(float d, float beta) {
  if (beta == 1.0f) return d;
  return powf(d, beta);
}
constexpr float kU32RelErr = 1.0f / 65536.0f;
// Relative separation below which two fp64 gaps count as a near-tie (about
// 64 ulp of the sum of the four u values involved).
constexpr double kTieRel = 1.0 / 281474976710656.0;  // 2^-48

struct SchedShared {
  int slot[kMaxEntries];
  long long first[kMaxEntries];
  long long span[kMaxEntries];
  long long mu2[kMaxEntries];  // 2*mu: mu is always a half-integer (midpoint of a contiguous span)
  int natoms[kMaxEntries];
  int ref[kMaxEntries][kMaxPassFrames + 1];
  float w[kMaxEntries][kMaxPassFrames + 1];
  float u32[kMaxEntries];
  double u64[kMaxEntries];   // fp64 u at the endpoints of the candidate pairs
  int dest[kMaxEntries];     // plan: destination index of a changed entry, -1 if unchanged
  int src0[kMaxEntries];     // plan: first source index of a changed entry
};

// Lowest (value, index) over the warp.
__device__ __forceinline__ void warp_argmin(double& v, int& i) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const double ov = __shfl_xor_sync(0xffffffffu, v, off);
    const int oi = __shfl_xor_sync(0xffffffffu, i, off);
    if (ov < v || (ov == v && oi < i)) { v = ov; i = oi; }
  }
}

// Algorithm S1 for `frames` units, one warp.  The pair chosen for each frame
// is exactly the argmin (lowest index on ties) of the fp64 gaps
// |warp_u(t - mu_{i+1}) - warp_u(t - mu_i)|: every pair is first scored in
// fp32 with an error bound E_i, and only pairs whose fp32 interval can reach
// the smallest upper bound U = min_k (g32_k + E_k) are scored again in fp64.
// A pair outside that set has a true gap above the true minimum by more than
// the fp64 rounding, so it cannot be the fp64 argmin either.
// Reads the entry table of `in` and writes the updated table and the pass's
// merge plan to `out` (the same state for an in-place pass, another buffer
// for a pass scheduled ahead of its frames).  Run by one full warp.
__device__ __noinline__ void schedule_pass(SchedShared& s, const DevState* in, DevState* out, unsigned int* status,
                                           int frames, int M, double beta, int anchor, int op, int expected_count) {
  const int lane = threadIdx.x & 31;
  const DevMeta& mi = in->meta;
  int count = mi.count;
  if (count != expected_count || count < 0 || count > M) {
    if (lane == 0) atomicOr(status, kStatusCountMismatch);
    if (lane == 0) { out->plan.n_src = 0; out->plan.near_tie_t = -1; }
    return;
  }
  const long long t0 = mi.t_next;
  const float beta32 = (float)beta;
  for (int i = lane; i < count; i += 32) {
    s.slot[i] = mi.slot[i];
    s.first[i] = mi.first[i];
    s.span[i] = mi.span[i];
    s.mu2[i] = __double2ll_rn(2.0 * mi.mu[i]);
    s.natoms[i] = 1;
    s.ref[i][0] = mi.slot[i];  // content: the block now stored in its own slot
    s.w[i][0] = 1.0f;
  }
  __syncwarp();
  int merged[kMaxPassFrames];
  long long near_tie = -1;  // first frame of the pass decided on a near-tie (lane 0)
  for (int f = 0; f < frames; ++f) {
    const long long t = t0 + f;
    if (lane == 0) {  // Append (K_t, V_t, t, 1)
      s.first[count] = t;
      s.span[count] = 1;
      s.mu2[count] = 2 * t;
      s.natoms[count] = 1;
      s.ref[count][0] = -(f + 1);
      s.w[count][0] = 1.0f;
      s.slot[count] = count;  // next free slot unless a merge frees one below
    }
    count += 1;
    __syncwarp();
    merged[f] = -1;
    if (kBoundsChecks && !index_ok(count - 1, kMaxEntries, status)) break;  // the append above stayed in the table
    if (count <= M) continue;

    // Eligible pairs: (i, i+1) for i <= count-3 (the pair holding the newest is excluded).
    const int npairs = count - 2;
    for (int i = lane; i <= npairs; i += 32) s.u32[i] = warp_u32(0.5f * (float)(2 * t - s.mu2[i]), beta32);
    __syncwarp();
    float ub = INFINITY;
    for (int i = lane; i < npairs; i += 32) {
      const float a = s.u32[i], b = s.u32[i + 1];
      ub = fminf(ub, fabsf(b - a) + kU32RelErr * (a + b));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ub = fminf(ub, __shfl_xor_sync(0xffffffffu, ub, off));
    // Candidates: pairs whose fp32 interval reaches ub (npairs < 64: one bit each).
    unsigned long long cm = 0;
    for (int i0 = 0; i0 < npairs; i0 += 32) {
      const int i = i0 + lane;
      bool cand = false;
      if (i < npairs) {
        const float a = s.u32[i], b = s.u32[i + 1];
        cand = fabsf(b - a) - kU32RelErr * (a + b) <= ub;
      }
      cm |= (unsigned long long)__ballot_sync(0xffffffffu, cand) << i0;
    }
    if (cm == 0) cm = (1ull << npairs) - 1;  // no finite bound (cannot happen for finite u): decide all in fp64
    int bi;
    if (__popcll(cm) == 1) {
      bi = __ffsll((long long)cm) - 1;  // the single candidate
    } else {
      // Several pairs may be the minimum: decide in fp64.  u is evaluated once
      // per endpoint of a candidate pair, one endpoint per lane (fp64 is slow
      // on this part, so the evaluations run side by side, not per pair).
      const unsigned long long em = cm | (cm << 1);
      const int nep = __popcll(em);
      for (int r0 = 0; r0 < nep; r0 += 32) {
        const int r = r0 + lane;
        if (r < nep) {
          unsigned long long m = em;
          for (int k = 0; k < r; ++k) m &= m - 1;  // drop the r lowest endpoints
          const int e = __ffsll((long long)m) - 1;
          s.u64[e] = warp_u(0.5 * (double)(2 * t - s.mu2[e]), beta);
        }
      }
      __syncwarp();
      double best = INFINITY;
      bi = 0x7fffffff;
      for (int i = lane; i < npairs; i += 32)
        if ((cm >> i) & 1) {
          const double g = fabs(s.u64[i + 1] - s.u64[i]);
          if (g < best) { best = g; bi = i; }
        }
      warp_argmin(best, bi);
      double second = INFINITY;
      int si = 0x7fffffff;
      for (int i = lane; i < npairs; i += 32)
        if (((cm >> i) & 1) && i != bi) {
          const double g = fabs(s.u64[i + 1] - s.u64[i]);
          if (g < second) { second = g; si = i; }
        }
      warp_argmin(second, si);
      // Certify the decision.  Any faithful fp64 d^beta (this one, or a host
      // libm's) is within a few ulp of the true value, so two gaps closer than
      // 2^-48 (u_b + u_b+1 + u_s + u_s+1) may be ordered differently by another
      // evaluation.  Exact evaluations settle every comparison the same way:
      // beta = 1 (u(d) = d) and beta = 0.5 where every u involved is an exact
      // square root.
      if (lane == 0 && si != 0x7fffffff) {
        const double ub0 = s.u64[bi], ub1 = s.u64[bi + 1], us0 = s.u64[si], us1 = s.u64[si + 1];
        bool exact = beta == 1.0;
        if (beta == 0.5) {
          exact = true;
          const int ix[4] = {bi, bi + 1, si, si + 1};
          for (int k = 0; k < 4; ++k) {
            const double u = s.u64[ix[k]];
            exact = exact && fma(u, u, -0.5 * (double)(2 * t - s.mu2[ix[k]])) == 0.0;
          }
        }
        if (!exact && second - best <= kTieRel * (ub0 + ub1 + us0 + us1) && near_tie < 0) near_tie = t;
      }
    }
    const int j = bi;
    if (kBoundsChecks && !index_ok(j, count - 2, status)) break;  // an eligible pair: j + 1 <= count - 2
    merged[f] = j;
    if (lane == 0) {
      const long long sa = s.span[j], sb = s.span[j + 1];
      const long long s_new = sa + sb;
      long long mu2_new;
      if (anchor && j == 0) {
        mu2_new = 0;  // the anchor keeps its block and centre
      } else {
        // mu_new = (s_j mu_j + s_{j+1} mu_{j+1}) / s_new, exactly, on 2*mu (the
        // span-weighted centre of two adjacent contiguous runs is a half-integer).
        mu2_new = (sa * s.mu2[j] + sb * s.mu2[j + 1]) / s_new;
        float wa = 1.0f, wb = 1.0f;
        if (op == FADEMEM_MERGE_WEIGHTED) {
          wa = sqrtf((float)sa) / (sqrtf((float)sa) + sqrtf((float)sb));
          wb = 1.0f - wa;
        } else if (op == FADEMEM_MERGE_AVERAGE) {
          wa = 0.5f; wb = 0.5f;
        } else if (op == FADEMEM_MERGE_SELECT_NEAREST) {
          wa = 0.0f; wb = 1.0f;
        }
        int n = 0;
        int ref[kMaxPassFrames + 1];
        float w[kMaxPassFrames + 1];
        for (int k = 0; k < s.natoms[j]; ++k)
          if (wa != 0.0f) { ref[n] = s.ref[j][k]; w[n] = s.w[j][k] * wa; ++n; }
        for (int k = 0; k < s.natoms[j + 1]; ++k)
          if (wb != 0.0f && n <= kMaxPassFrames) { ref[n] = s.ref[j + 1][k]; w[n] = s.w[j + 1][k] * wb; ++n; }
        s.natoms[j] = n;
        for (int k = 0; k < n; ++k) { s.ref[j][k] = ref[k]; s.w[j][k] = w[k]; }
      }
      s.span[j] = s_new;
      s.mu2[j] = mu2_new;
    }
    const int freed = s.slot[j + 1];
    __syncwarp();
    // Remove m_{j+1}: entries j+2 .. count-1 move down one place (lane-parallel).
    for (int base = j + 1; base < count - 1; base += 32) {
      const int i = base + lane;
      int slot = 0, na = 0;
      long long first = 0, span = 0, mu2 = 0;
      int ref[kMaxPassFrames + 1];
      float w[kMaxPassFrames + 1];
      const bool mv = i < count - 1;
      if (mv) {
        slot = s.slot[i + 1]; first = s.first[i + 1]; span = s.span[i + 1]; mu2 = s.mu2[i + 1];
        na = s.natoms[i + 1];
#pragma unroll
        for (int k = 0; k <= kMaxPassFrames; ++k) { ref[k] = s.ref[i + 1][k]; w[k] = s.w[i + 1][k]; }
      }
      __syncwarp();
      if (mv) {
        s.slot[i] = slot; s.first[i] = first; s.span[i] = span; s.mu2[i] = mu2; s.natoms[i] = na;
#pragma unroll
        for (int k = 0; k <= kMaxPassFrames; ++k) { s.ref[i][k] = ref[k]; s.w[i][k] = w[k]; }
      }
      __syncwarp();
    }
    if (lane == 0) s.slot[count - 2] = freed;  // the newest entry takes m_{j+1}'s slot
    count -= 1;
    __syncwarp();
  }

  // Merge plan: every entry whose block changed becomes a destination; its
  // sources are stored contiguously, in entry order (lane-parallel prefix sums).
  int nd = 0, ns = 0;
  for (int base = 0; base < count; base += 32) {
    const int i = base + lane;
    bool changed = false;
    int na = 0;
    if (i < count) {
      changed = !(s.natoms[i] == 1 && s.ref[i][0] == s.slot[i] && s.w[i][0] == 1.0f);
      na = changed ? s.natoms[i] : 0;
    }
    const unsigned cm = __ballot_sync(0xffffffffu, changed);
    int incl = na;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += o;
    }
    if (i < count) {
      s.dest[i] = changed ? nd + __popc(cm & ((1u << lane) - 1u)) : -1;
      s.src0[i] = ns + incl - na;
    }
    nd += __popc(cm);
    ns += __shfl_sync(0xffffffffu, incl, 31);
  }
  __syncwarp();
  __syncwarp();  // every lane has read `in` before `out` (possibly the same) is written
  DevPlan& p = out->plan;
  DevMeta& m = out->meta;
  const bool overflow = nd > kMaxDest || ns > kMaxSrc;
  if (!overflow) {
    for (int i = lane; i < count; i += 32) {
      const int d = s.dest[i];
      if (d < 0) continue;
      if (kBoundsChecks && !index_ok(d, kMaxDest, status)) continue;
      p.dest_slot[d] = s.slot[i];
      for (int k = 0; k < s.natoms[i]; ++k) {
        const int q = s.src0[i] + k;
        if (kBoundsChecks && !index_ok(q, kMaxSrc, status)) break;
        p.src_ref[q] = s.ref[i][k];
        p.src_w[q] = s.w[i][k];
        p.src_dest[q] = d;
      }
    }
  }
  if (lane == 0) {
    if (overflow) { nd = 0; ns = 0; atomicOr(status, kStatusPlanOverflow); }
    p.n_src = ns;
    p.n_dest = nd;
    p.frames = frames;
    p.op = op;
    p.near_tie_t = near_tie;
    for (int f = 0; f < kMaxPassFrames; ++f) p.merged_pair[f] = f < frames ? merged[f] : -1;
    m.count = count;
    m.t_next = t0 + frames;
  }
  for (int i = lane; i < count; i += 32) {
    m.slot[i] = s.slot[i];
    m.first[i] = s.first[i];
    m.span[i] = s.span[i];
    m.mu[i] = 0.5 * (double)s.mu2[i];
  }
}

__global__ void __launch_bounds__(32) schedule_kernel(const DevState* in, DevState* out, unsigned int* status,
                                                      int frames, int M, double beta, int anchor, int op,
                                                      int expected_count) {
  __shared__ SchedShared s;
  // The consolidation kernel launched after this one may start now: it waits
  // for this grid's completion before it reads the plan.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  schedule_pass(s, in, out, status, frames, M, beta, anchor, op, expected_count);
}

// ---- K2 ------------------------------------------------------------------

template <typename T> struct Vec;
template <> struct Vec<float> {
  static constexpr int kN = 4;
  __device__ static void unpack(const uint4& v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
  __device__ static uint4 pack(const float* f) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]), __float_as_uint(f[3]));
  }
};
template <> struct Vec<__nv_bfloat16> {
  static constexpr int kN = 8;
  __device__ static void unpack(const uint4& v, float* f) {
    const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
  __device__ static uint4 pack(const float* f) {
    unsigned w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __nv_bfloat162 b = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);  // .x -> low half
      w[i] = *reinterpret_cast<unsigned*>(&b);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
};

struct ConsolidateArgs {
  char* cache;            // workspace cache base
  size_t cache_bytes;     // every layer's memory, from cache (bounds checks)
  size_t frame_bytes;     // one layer's K (or V) frames of the pass (bounds checks)
  const DevState* st;
  int L, H, M, N, D;
  int dv_shift;           // log2(D / elements per vector)
  size_t slab_elems;      // N * D
  size_t kv_elems;        // H * M * N * D
  size_t layer_elems;     // stride between layers, in elements
  // Lookahead: block 0 of the grid schedules the next pass of la_frames units
  // from la_in's entry table into la_out (skipped if null).
  const DevState* la_in;
  DevState* la_out;
  unsigned int* status;
  unsigned long long* totals;  // [blocks moved, passes] since the memory was created
  int la_frames, la_expected, la_anchor, la_op;
  double la_beta;
  int bx;                 // blocks per (layer, K|V, head) row
  // Temporal RoPE: K frame sources of the pass are rotated by -(t0 + f) omega_k
  // on their first rope_pairs complex pairs as they are loaded.
  int rope_pairs;
  long long rope_t0;
  double rope_omega[kMaxRopePairs];
  PassSources srcs;
};

// (cos a, sin a) of a = position * omega in fp32, with the angle reduced to
// [-pi, pi] in fp64 first: positions reach tens of thousands of frames, far
// beyond where an fp32 angle keeps its precision.
__device__ __forceinline__ float2 rope_cos_sin(double position, double omega) {
  const double two_pi = 6.283185307179586476925;
  double ang = position * omega;
  ang -= two_pi * rint(ang / two_pi);
  float sn, cs;
  sincosf((float)ang, &sn, &cs);
  return make_float2(cs, sn);
}

// Rotate the complex pairs of one 16-byte vector (x[2e], x[2e+1]; pair index
// pair0 + e) that lie in the temporal band (pair < P), by the table cs[pair].
template <int kN>
__device__ __forceinline__ void rope_rotate_vec(float* x, int pair0, int P, const float2* cs) {
#pragma unroll
  for (int e = 0; e < kN / 2; ++e) {
    if (pair0 + e < P) {
      const float2 r = cs[pair0 + e];
      const float x0 = x[2 * e], x1 = x[2 * e + 1];
      x[2 * e] = x0 * r.x - x1 * r.y;
      x[2 * e + 1] = x0 * r.y + x1 * r.x;
    }
  }
}

// K2 geometry: one wave of 256-thread blocks, 4 per SM (64 registers a
// thread), spread over the (layer, K|V, head) rows.  Each thread owns one
// 16-byte vector coordinate per iteration: it loads every plan source at that
// coordinate (all loads in flight together), then combines and stores every
// destination.  Because each read of a coordinate precedes every write to it
// in the same thread, slots that are both read and rewritten need no second
// buffer.  kNS bounds the sources of the pass: F frames make at most F merges,
// which touch at most 2F entries, plus F frame copies, so kNS = 3F suffices;
// a larger plan is refused through the status word.
constexpr int kConsThreads = 256;
// Resident blocks per SM: 4 (64 registers) while the sources fit, 3 for 12
// sources or with the RoPE rotation.
__host__ __device__ constexpr int cons_blocks_per_sm(int ns_max, bool rope) { return ns_max <= 9 && !rope ? 4 : 3; }
// Vectors a thread handles in a consolidation with more rows than one wave
// holds (each row is then split into blocks of this many vectors a thread).
constexpr int kConsShortIters = 4;

template <typename T, bool kMax, int kNS, bool kRope>
__global__ void __launch_bounds__(kConsThreads, cons_blocks_per_sm(kNS, kRope)) consolidate_kernel(
    const __grid_constant__ ConsolidateArgs a) {
  using V = Vec<T>;
  __shared__ const T* s_base[kMaxSrc];  // source k at token n: s_base[k] + n * (token stride) + d
  __shared__ T* s_dst[kMaxSrc];         // destination of the run that source k ends
  __shared__ float s_w[kMaxSrc];
  __shared__ unsigned s_frame_mask, s_end_mask;  // bit k: source k is a frame / ends its run
  __shared__ int s_ns;
  __shared__ int s_frame_of[kMaxSrc];                      // frame index f of a frame source
  __shared__ float2 s_rope_cs[kRope ? kMaxPassFrames : 1][kRope ? kMaxRopePairs : 1];  // by -(t0 + f) omega_k
  // Launched as a programmatic dependent of the schedule kernel: wait for it
  // (and every earlier grid of the stream) before reading any global memory.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (blockIdx.x == 0) {
    // Schedule the next pass while the other blocks apply this one: it reads
    // the entry table this pass already produced and writes the other buffer.
    // Block 0 is dispatched first, so the schedule overlaps the whole copy.
    __shared__ SchedShared sched;
    if (a.la_out != nullptr && threadIdx.x < 32)
      schedule_pass(sched, a.la_in, a.la_out, a.status, a.la_frames, a.M, a.la_beta, a.la_anchor, a.la_op,
                    a.la_expected);
    return;
  }
  const int bx = (int)(blockIdx.x - 1) % a.bx;    // block within its row
  const int slab = (int)(blockIdx.x - 1) / a.bx;  // row: (l * 2 + kv) * H + h
  const int h = slab % a.H;
  const int kv = (slab / a.H) & 1;
  const int l = slab / (2 * a.H);
  T* cache = reinterpret_cast<T*>(a.cache) + (size_t)l * a.layer_elems + (size_t)kv * a.kv_elems +
             (size_t)h * a.M * a.slab_elems;
  if (threadIdx.x < 32) {
    // The plan lists the sources of each changed slot consecutively; lane k
    // decodes source k (all lanes at once, no dependent chain of loads).
    const DevPlan& p = a.st->plan;
    const int k = threadIdx.x;
    int ns = p.n_src;
    if (ns < 0 || ns > kMaxSrc) ns = kMaxSrc + 1;  // refused below (ns > kNS)
    bool frame = false, end = false, bad = false;
    if (k < ns && k < kMaxSrc) {
      int r = p.src_ref[k];
      int dk = p.src_dest[k];
      if (dk < 0 || dk >= kMaxDest || r >= a.M || r < -kMaxPassFrames || p.dest_slot[dk] < 0 ||
          p.dest_slot[dk] >= a.M) {
        bad = true;
        dk = 0;
        r = 0;
      }
      frame = r < 0;
      end = (k + 1 == ns) || (k + 1 < kMaxSrc && p.src_dest[k + 1] != dk);
      s_base[k] = frame ? reinterpret_cast<const T*>(a.srcs.src[l][kv]) + (size_t)(-r - 1) * a.N * a.H * a.D +
                              (size_t)h * a.D
                        : cache + (size_t)r * a.slab_elems;
      s_w[k] = p.src_w[k];
      s_dst[k] = cache + (size_t)(bad ? 0 : p.dest_slot[dk]) * a.slab_elems;
      s_frame_of[k] = frame ? -r - 1 : 0;
    }
    const unsigned fm = __ballot_sync(0xffffffffu, frame), em = __ballot_sync(0xffffffffu, end);
    if (__any_sync(0xffffffffu, bad)) ns = kMaxSrc + 1;
    if (k == 0) {
      s_frame_mask = fm;
      s_end_mask = em;
      s_ns = ns;
      if (blockIdx.x == 1) {
        atomicAdd(&a.totals[0], (unsigned long long)(p.n_src + p.n_dest));  // per layer, K and V
        atomicAdd(&a.totals[1], 1ull);
        // A decision of this pass that the schedule could not certify: report
        // it (first frame kept) now that the pass is applied.
        const long long nt = p.near_tie_t;
        if (nt >= 0) {
          atomicOr(a.status, kStatusNearTie);
          atomicCAS(reinterpret_cast<unsigned long long*>(reinterpret_cast<char*>(a.status) + kNearTieFrameOffset),
                    0ull, (unsigned long long)(nt + 1));
        }
      }
    }
  }
  // Temporal RoPE: the K rows of this pass's frames lose their phase.
  const bool rope = kRope && kv == 0;
  if (kRope && rope) {
    for (int t = threadIdx.x; t < kMaxPassFrames * a.rope_pairs; t += blockDim.x) {
      const int f = t / a.rope_pairs, k = t % a.rope_pairs;
      s_rope_cs[f][k] = rope_cos_sin(-(double)(a.rope_t0 + f), a.rope_omega[k]);
    }
  }
  __syncthreads();
  const int ns = s_ns;
  if (ns == 0) return;
  if (ns > kNS) {
    if (threadIdx.x == 0 && blockIdx.x == 1) atomicOr(a.status, kStatusPlanOverflow);
    return;
  }
  const unsigned fmask = s_frame_mask, emask = s_end_mask;
  const int dvmask = (1 << a.dv_shift) - 1;
  const int nvec = a.N << a.dv_shift;
  const unsigned frame_tok = (unsigned)(a.H * a.D);

  // Offsets within one slab (< N*D) or one frame (< N*H*D < 2^31) fit in 32 bits.
  for (int v = bx * kConsThreads + threadIdx.x; v < nvec; v += a.bx * kConsThreads) {
    const unsigned n = (unsigned)v >> a.dv_shift;
    const unsigned d = (unsigned)(v & dvmask) * V::kN;
    const unsigned off_slab = n * (unsigned)a.D + d;
    const unsigned off_frame = n * frame_tok + d;
    uint4 raw[kNS];
#pragma unroll
    for (int k = 0; k < kNS; ++k)
      if (k < ns) {
        const bool fr = (fmask >> k) & 1;
        const T* src = s_base[k] + (fr ? off_frame : off_slab);
        if (kBoundsChecks && !bounds_ok(fr ? dev_range(a.srcs.src[l][kv], a.frame_bytes)
                                           : dev_range(a.cache, a.cache_bytes),
                                        src, sizeof(uint4), a.status)) {
          raw[k] = make_uint4(0u, 0u, 0u, 0u);
          continue;
        }
        raw[k] = __ldcs(reinterpret_cast<const uint4*>(src));
      }
    float acc[V::kN];
#pragma unroll
    for (int e = 0; e < V::kN; ++e) acc[e] = kMax ? -INFINITY : 0.f;
#pragma unroll
    for (int k = 0; k < kNS; ++k) {
      if (k < ns) {
        float x[V::kN];
        V::unpack(raw[k], x);
        if (kRope && rope && ((fmask >> k) & 1) && (int)d < 2 * a.rope_pairs)
          rope_rotate_vec<V::kN>(x, (int)d / 2, a.rope_pairs, s_rope_cs[s_frame_of[k]]);
        const float w = s_w[k];
#pragma unroll
        for (int e = 0; e < V::kN; ++e) acc[e] = kMax ? fmaxf(acc[e], x[e]) : fmaf(w, x[e], acc[e]);
        if ((emask >> k) & 1) {
          T* dst = s_dst[k] + off_slab;
          if (!kBoundsChecks || bounds_ok(dev_range(a.cache, a.cache_bytes), dst, sizeof(uint4), a.status))
            *reinterpret_cast<uint4*>(dst) = V::pack(acc);
#pragma unroll
          for (int e = 0; e < V::kN; ++e) acc[e] = kMax ? -INFINITY : 0.f;
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_schedule(const DevState* in, DevState* out, unsigned int* status, int frames, int M, double beta,
                            int anchor, int op, int expected_count, cudaStream_t stream) {
  if (frames < 1 || frames > kMaxPassFrames) return cudaErrorInvalidValue;
  schedule_kernel<<<1, 32, 0, stream>>>(in, out, status, frames, M, beta, anchor, op, expected_count);
  return cudaGetLastError();
}

cudaError_t launch_consolidate(const Geometry& g, void* cache_base, const DevState* st, const PassSources& srcs,
                               int frames, int op, const Lookahead& la, const PassRope& rope,
                               cudaStream_t stream) {
  static_assert(kMaxSrc == 3 * kMaxPassFrames, "a pass of F frames has at most 3F sources");
  ConsolidateArgs a;
  a.la_in = la.in;
  a.la_out = la.out;
  a.status = la.status;
  a.totals = la.totals;
  a.la_frames = la.frames;
  a.la_expected = la.expected_count;
  a.la_anchor = la.anchor;
  a.la_op = la.op;
  a.la_beta = la.beta;
  a.rope_pairs = rope.pairs;
  a.rope_t0 = rope.t0;
  for (int k = 0; k < kMaxRopePairs; ++k) a.rope_omega[k] = rope.omega[k];
  a.cache = reinterpret_cast<char*>(cache_base);
  a.cache_bytes = (size_t)g.L * g.layer_bytes;
  a.frame_bytes = (size_t)frames * g.N * g.H * g.D * g.elem;
  a.st = st;
  a.L = g.L; a.H = g.H; a.M = g.M; a.N = g.N; a.D = g.D;
  const int per_vec = g.dtype == FADEMEM_BF16 ? 8 : 4;
  int dv = g.D / per_vec, shift = 0;
  while ((1 << shift) < dv) ++shift;
  a.dv_shift = shift;
  a.slab_elems = g.slab_elems;
  a.kv_elems = g.kv_elems;
  a.layer_elems = g.layer_bytes / g.elem;
  a.srcs = srcs;
  const int nvec = g.N * dv;
  // While the layer*K|V*head rows fit in one wave (SMs x resident blocks), that
  // wave is spread evenly over them and each thread strides over its row's
  // vectors.  More rows than that (a memory of many layers) would end in a
  // partial wave of whole rows, too few blocks to keep HBM busy while they
  // stream their rows (a 30-layer consolidation ran at 82% of the copy peak
  // so); there each row is cut into short blocks of kConsShortIters vectors a
  // thread, and the last of many short waves ends with the others (97%).
  const int num_sms = current_device_sm_count(148);
  const int nsb = frames <= 2 ? 0 : frames == 3 ? 1 : 2;  // sources <= 3F: 6, 9 or 12
  const int rows = g.L * 2 * g.H;
  const int wave = num_sms * cons_blocks_per_sm(6 + 3 * nsb, rope.pairs > 0) - 1;  // - 1: the lookahead block
  int bx = rows <= wave ? wave / rows : (nvec + kConsThreads * kConsShortIters - 1) / (kConsThreads * kConsShortIters);
  const int bx_max = (nvec + kConsThreads - 1) / kConsThreads;
  if (bx > bx_max) bx = bx_max;
  if (bx < 1) bx = 1;
  a.bx = bx;
  dim3 grid(1 + bx * rows);  // block 0: the lookahead schedule
  const bool mx = op == FADEMEM_MERGE_MAX_POOL;
  using Kern = void (*)(const ConsolidateArgs);
#define FM_K2(T, MX, R) {consolidate_kernel<T, MX, 6, R>, consolidate_kernel<T, MX, 9, R>, consolidate_kernel<T, MX, 12, R>}
  static const Kern kerns[2][2][2][3] = {
      {{FM_K2(float, false, false), FM_K2(float, true, false)},
       {FM_K2(__nv_bfloat16, false, false), FM_K2(__nv_bfloat16, true, false)}},
      {{FM_K2(float, false, true), FM_K2(float, true, true)},
       {FM_K2(__nv_bfloat16, false, true), FM_K2(__nv_bfloat16, true, true)}}};
#undef FM_K2
  const Kern kern = kerns[rope.pairs > 0 ? 1 : 0][g.dtype == FADEMEM_BF16 ? 1 : 0][mx ? 1 : 0][nsb];
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kConsThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}


// ---- K2b: temporal RoPE re-index ------------------------------------------

namespace {

struct RephaseArgs {
  char* cache;
  size_t cache_bytes;  // every layer's memory, from cache (bounds checks)
  unsigned int* status;
  const DevState* st;
  int H, M, N, D, count, bx, dv_shift, pairs;
  long long t_next;
  size_t slab_elems, kv_elems, layer_elems;
  double omega[kMaxRopePairs];
};

// One wave of 256-thread blocks over the (layer, head, entry) rows; block x of
// a row streams 16-byte vectors of the entry's stored K slab to the same place
// in the K_att block, rotating the vectors of the temporal band.  Four loads
// are in flight per thread.  HBM-bound: count * N * D * elem read and written
// per (layer, head).
template <typename T>
__global__ void __launch_bounds__(256) rephase_kernel(const __grid_constant__ RephaseArgs a) {
  using V = Vec<T>;
  __shared__ float2 s_cs[kMaxRopePairs];
  const int bx = (int)blockIdx.x % a.bx;
  const int row = (int)blockIdx.x / a.bx;
  const int i = row % a.count;
  const int h = (row / a.count) % a.H;
  const int l = row / (a.count * a.H);
  int slot = a.st->meta.slot[i];
  if (slot < 0 || slot >= a.M) {  // not a valid table (refused earlier by the schedule checks)
    if (kBoundsChecks && threadIdx.x == 0) atomicOr(a.status, kStatusBounds);
    return;
  }
  const double tau = (double)(a.t_next - a.count + i);  // re-indexed position of entry i
  for (int k = threadIdx.x; k < a.pairs; k += blockDim.x) s_cs[k] = rope_cos_sin(tau, a.omega[k]);
  __syncthreads();
  const T* src = reinterpret_cast<const T*>(a.cache) + (size_t)l * a.layer_elems + (size_t)h * a.M * a.slab_elems +
                 (size_t)slot * a.slab_elems;
  T* dst = const_cast<T*>(src) + 2 * a.kv_elems;  // K_att follows K and V
  const int nvec = a.N << a.dv_shift;
  const int dvmask = (1 << a.dv_shift) - 1;
  const int step = a.bx * blockDim.x;
  constexpr int kU = 4;
  for (int v0 = bx * blockDim.x + threadIdx.x; v0 < nvec; v0 += kU * step) {
    uint4 raw[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int v = v0 + u * step;
      if (v < nvec) {
        if (kBoundsChecks && !bounds_ok(dev_range(a.cache, a.cache_bytes), reinterpret_cast<const uint4*>(src) + v,
                                        sizeof(uint4), a.status)) {
          raw[u] = make_uint4(0u, 0u, 0u, 0u);
          continue;
        }
        raw[u] = __ldcs(reinterpret_cast<const uint4*>(src) + v);
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int v = v0 + u * step;
      if (v >= nvec) continue;
      const int d = (v & dvmask) * V::kN;
      uint4 w = raw[u];
      if (d < 2 * a.pairs) {
        float x[V::kN];
        V::unpack(w, x);
        rope_rotate_vec<V::kN>(x, d / 2, a.pairs, s_cs);
        w = V::pack(x);
      }
      if (kBoundsChecks &&
          !bounds_ok(dev_range(a.cache, a.cache_bytes), reinterpret_cast<uint4*>(dst) + v, sizeof(uint4), a.status))
        continue;
      reinterpret_cast<uint4*>(dst)[v] = w;
    }
  }
}

}  // namespace

cudaError_t launch_rephase(const Geometry& g, void* cache_base, const DevState* st, int count, long long t_next,
                           unsigned int* status, cudaStream_t stream) {
  if (count <= 0 || g.rope_pairs <= 0) return cudaSuccess;
  RephaseArgs a;
  a.cache = reinterpret_cast<char*>(cache_base);
  a.cache_bytes = (size_t)g.L * g.layer_bytes;
  a.status = status;
  a.st = st;
  a.H = g.H; a.M = g.M; a.N = g.N; a.D = g.D;
  a.count = count;
  a.pairs = g.rope_pairs;
  a.t_next = t_next;
  a.slab_elems = g.slab_elems;
  a.kv_elems = g.kv_elems;
  a.layer_elems = g.layer_bytes / g.elem;
  for (int k = 0; k < kMaxRopePairs; ++k) a.omega[k] = g.rope_omega[k];
  const int per_vec = g.dtype == FADEMEM_BF16 ? 8 : 4;
  int dv = g.D / per_vec, shift = 0;
  while ((1 << shift) < dv) ++shift;
  a.dv_shift = shift;
  const int num_sms = current_device_sm_count(148);
  const long long rows = (long long)g.L * g.H * count;
  const int nvec = g.N * dv;
  long long bx = (long long)num_sms * 8 / rows;  // one wave of 8 resident blocks per SM
  const long long bx_max = (nvec + 255) / 256;
  if (bx > bx_max) bx = bx_max;
  if (bx < 1) bx = 1;
  a.bx = (int)bx;
  const dim3 grid((unsigned)(bx * rows));
  if (g.dtype == FADEMEM_BF16)
    rephase_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(a);
  else
    rephase_kernel<float><<<grid, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

int current_device_sm_count(int fallback) {
  static PerDevice<int> table;
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return fallback;
  const bool ok = table.get(dev, [](int d, int* v) {
    return cudaDeviceGetAttribute(v, cudaDevAttrMultiProcessorCount, d) == cudaSuccess && *v > 0;
  }, &n);
  return ok ? n : fallback;
}

}  // namespace fademem
