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

struct SchedShared {
  int slot[kMaxEntries];
  long long first[kMaxEntries];
  long long span[kMaxEntries];
  double mu[kMaxEntries];
  int natoms[kMaxEntries];
  int ref[kMaxEntries][kMaxPassFrames + 1];
  double w[kMaxEntries][kMaxPassFrames + 1];
};

__global__ void __launch_bounds__(32) schedule_kernel(DevState* st, int frames, int M, double beta, int anchor,
                                                      int op, int expected_count) {
  __shared__ SchedShared s;
  const int lane = threadIdx.x;
  DevMeta& m = st->meta;
  int count = m.count;
  if (count != expected_count || count < 0 || count > M) {
    if (lane == 0) atomicOr(&st->status, kStatusCountMismatch);
    if (lane == 0) st->plan.n_src = 0;
    return;
  }
  const long long t0 = m.t_next;
  for (int i = lane; i < count; i += 32) {
    s.slot[i] = m.slot[i];
    s.first[i] = m.first[i];
    s.span[i] = m.span[i];
    s.mu[i] = m.mu[i];
    s.natoms[i] = 1;
    s.ref[i][0] = m.slot[i];  // content: the block now stored in its own slot
    s.w[i][0] = 1.0;
  }
  __syncwarp();
  int merged[kMaxPassFrames];
  for (int f = 0; f < frames; ++f) {
    const long long t = t0 + f;
    if (lane == 0) {  // Append (K_t, V_t, t, 1)
      s.first[count] = t;
      s.span[count] = 1;
      s.mu[count] = (double)t;
      s.natoms[count] = 1;
      s.ref[count][0] = -(f + 1);
      s.w[count][0] = 1.0;
      s.slot[count] = count;  // next free slot unless a merge frees one below
    }
    count += 1;
    __syncwarp();
    merged[f] = -1;
    if (count <= M) continue;

    // Eligible pairs: (i, i+1) for i <= count-3 (the pair holding the newest is excluded).
    const int npairs = count - 2;
    double best = INFINITY;
    int bi = 0x7fffffff;
    for (int i = lane; i < npairs; i += 32) {
      const double g = fabs(warp_u((double)t - s.mu[i + 1], beta) - warp_u((double)t - s.mu[i], beta));
      if (g < best) { best = g; bi = i; }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const double og = __shfl_xor_sync(0xffffffffu, best, off);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
      if (og < best || (og == best && oi < bi)) { best = og; bi = oi; }
    }
    const int j = bi;
    merged[f] = j;
    if (lane == 0) {
      const long long sa = s.span[j], sb = s.span[j + 1];
      const long long s_new = sa + sb;
      double mu_new;
      if (anchor && j == 0) {
        mu_new = 0.0;  // the anchor keeps its block and centre
      } else {
        mu_new = ((double)sa * s.mu[j] + (double)sb * s.mu[j + 1]) / (double)s_new;
        double wa = 1.0, wb = 1.0;
        if (op == FADEMEM_MERGE_WEIGHTED) {
          wa = sqrt((double)sa) / (sqrt((double)sa) + sqrt((double)sb));
          wb = 1.0 - wa;
        } else if (op == FADEMEM_MERGE_AVERAGE) {
          wa = 0.5; wb = 0.5;
        } else if (op == FADEMEM_MERGE_SELECT_NEAREST) {
          wa = 0.0; wb = 1.0;
        }
        int n = 0;
        int ref[kMaxPassFrames + 1];
        double w[kMaxPassFrames + 1];
        for (int k = 0; k < s.natoms[j]; ++k)
          if (wa != 0.0) { ref[n] = s.ref[j][k]; w[n] = s.w[j][k] * wa; ++n; }
        for (int k = 0; k < s.natoms[j + 1]; ++k)
          if (wb != 0.0 && n <= kMaxPassFrames) { ref[n] = s.ref[j + 1][k]; w[n] = s.w[j + 1][k] * wb; ++n; }
        s.natoms[j] = n;
        for (int k = 0; k < n; ++k) { s.ref[j][k] = ref[k]; s.w[j][k] = w[k]; }
      }
      s.span[j] = s_new;
      s.mu[j] = mu_new;
      const int freed = s.slot[j + 1];
      for (int i = j + 1; i < count - 1; ++i) {
        s.slot[i] = s.slot[i + 1];
        s.first[i] = s.first[i + 1];
        s.span[i] = s.span[i + 1];
        s.mu[i] = s.mu[i + 1];
        s.natoms[i] = s.natoms[i + 1];
        for (int k = 0; k < s.natoms[i]; ++k) { s.ref[i][k] = s.ref[i + 1][k]; s.w[i][k] = s.w[i + 1][k]; }
      }
      s.slot[count - 2] = freed;  // the newest entry takes m_{j+1}'s slot
    }
    count -= 1;
    __syncwarp();
  }

  if (lane == 0) {
    DevPlan& p = st->plan;
    int ns = 0, nd = 0;
    bool overflow = false;
    for (int i = 0; i < count; ++i) {
      const bool same = s.natoms[i] == 1 && s.ref[i][0] == s.slot[i] && s.w[i][0] == 1.0;
      if (same) continue;
      if (nd >= kMaxDest || ns + s.natoms[i] > kMaxSrc) { overflow = true; break; }
      p.dest_slot[nd] = s.slot[i];
      for (int k = 0; k < s.natoms[i]; ++k) {
        p.src_ref[ns] = s.ref[i][k];
        p.src_w[ns] = (float)s.w[i][k];
        p.src_dest[ns] = nd;
        ++ns;
      }
      ++nd;
    }
    if (overflow) { ns = 0; nd = 0; atomicOr(&st->status, kStatusPlanOverflow); }
    p.n_src = ns;
    p.n_dest = nd;
    p.frames = frames;
    p.op = op;
    for (int f = 0; f < kMaxPassFrames; ++f) p.merged_pair[f] = f < frames ? merged[f] : -1;
    m.count = count;
    m.t_next = t0 + frames;
  }
  for (int i = lane; i < count; i += 32) {
    m.slot[i] = s.slot[i];
    m.first[i] = s.first[i];
    m.span[i] = s.span[i];
    m.mu[i] = s.mu[i];
  }
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
  const DevState* st;
  int L, H, M, N, D;
  int dv_shift;           // log2(D / elements per vector)
  size_t slab_elems;      // N * D
  size_t kv_elems;        // H * M * N * D
  size_t layer_elems;     // stride between layers, in elements
  PassSources srcs;
};

template <typename T, bool kMax>
__global__ void __launch_bounds__(256) consolidate_kernel(const __grid_constant__ ConsolidateArgs a) {
  using V = Vec<T>;
  __shared__ int s_ref[kMaxSrc], s_dest[kMaxSrc], s_dslot[kMaxDest];
  __shared__ float s_w[kMaxSrc];
  __shared__ int s_ns;
  const DevPlan& p = a.st->plan;
  if (threadIdx.x < kMaxSrc) {
    s_ref[threadIdx.x] = p.src_ref[threadIdx.x];
    s_dest[threadIdx.x] = p.src_dest[threadIdx.x];
    s_w[threadIdx.x] = p.src_w[threadIdx.x];
  }
  if (threadIdx.x < kMaxDest) s_dslot[threadIdx.x] = p.dest_slot[threadIdx.x];
  if (threadIdx.x == 0) s_ns = p.n_src;
  __syncthreads();
  const int ns = s_ns;
  if (ns == 0) return;

  const int slab = blockIdx.y;  // (l * 2 + kv) * H + h
  const int h = slab % a.H;
  const int kv = (slab / a.H) & 1;
  const int l = slab / (2 * a.H);
  T* cache = reinterpret_cast<T*>(a.cache) + (size_t)l * a.layer_elems + (size_t)kv * a.kv_elems +
             (size_t)h * a.M * a.slab_elems;
  const T* frame0 = reinterpret_cast<const T*>(a.srcs.src[l][kv]);
  const size_t frame_elems = (size_t)a.N * a.H * a.D;
  const int dvmask = (1 << a.dv_shift) - 1;
  const int nvec = a.N << a.dv_shift;

  for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < nvec; v += gridDim.x * blockDim.x) {
    const int n = v >> a.dv_shift;
    const int d = (v & dvmask) * V::kN;
    const size_t in_slab = (size_t)n * a.D + d;
    const size_t in_frame = ((size_t)n * a.H + h) * a.D + d;
    uint4 raw[kMaxSrc];
#pragma unroll
    for (int k = 0; k < kMaxSrc; ++k) {
      if (k < ns) {
        const int r = s_ref[k];
        const T* src = r >= 0 ? cache + (size_t)r * a.slab_elems + in_slab
                              : frame0 + (size_t)(-r - 1) * frame_elems + in_frame;
        raw[k] = __ldcs(reinterpret_cast<const uint4*>(src));
      }
    }
    float acc[V::kN];
#pragma unroll
    for (int k = 0; k < kMaxSrc; ++k) {
      if (k < ns) {
        float x[V::kN];
        V::unpack(raw[k], x);
        const bool first = (k == 0) || (s_dest[k - 1] != s_dest[k]);
        const float w = s_w[k];
#pragma unroll
        for (int e = 0; e < V::kN; ++e) {
          if (kMax) acc[e] = first ? x[e] : fmaxf(acc[e], x[e]);
          else acc[e] = first ? w * x[e] : fmaf(w, x[e], acc[e]);
        }
        const bool last = (k + 1 == ns) || (s_dest[k + 1] != s_dest[k]);
        if (last) {
          T* dst = cache + (size_t)s_dslot[s_dest[k]] * a.slab_elems + in_slab;
          *reinterpret_cast<uint4*>(dst) = V::pack(acc);
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_schedule(DevState* st, int frames, int M, double beta, int anchor, int op, int expected_count,
                            cudaStream_t stream) {
  if (frames < 1 || frames > kMaxPassFrames) return cudaErrorInvalidValue;
  schedule_kernel<<<1, 32, 0, stream>>>(st, frames, M, beta, anchor, op, expected_count);
  return cudaGetLastError();
}

cudaError_t launch_consolidate(const Geometry& g, void* cache_base, const DevState* st, const PassSources& srcs,
                               int frames, int op, cudaStream_t stream) {
  (void)frames;
  ConsolidateArgs a;
  a.cache = reinterpret_cast<char*>(cache_base);
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
  const int threads = 256;
  int bx = (nvec + threads * 2 - 1) / (threads * 2);
  if (bx < 1) bx = 1;
  dim3 grid(bx, g.L * 2 * g.H);
  const bool mx = op == FADEMEM_MERGE_MAX_POOL;
  if (g.dtype == FADEMEM_BF16) {
    if (mx) consolidate_kernel<__nv_bfloat16, true><<<grid, threads, 0, stream>>>(a);
    else consolidate_kernel<__nv_bfloat16, false><<<grid, threads, 0, stream>>>(a);
  } else {
    if (mx) consolidate_kernel<float, true><<<grid, threads, 0, stream>>>(a);
    else consolidate_kernel<float, false><<<grid, threads, 0, stream>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace fademem
