// fp32 attention of query tokens over the memory (Sec. 3.3 last paragraph:
// the memory is the cached context the backbone's attention sees).
// Exact-precision path for the fp32 storage dtype: fp32 FMAs throughout (tf32
// tensor cores would not meet a 1e-5 relative tolerance), online softmax in
// the exp2 domain.
//
// One block of 128 threads computes a tile of 64 queries of one head.  Tiles
// of 32 keys are staged in shared memory by cp.async, double-buffered (the
// next tile loads while this one is used).  Per tile:
//   scores:  thread t holds a 4 x 4 block of S (queries t/8 + 16r, keys
//            t%8 + 8i), dot products over the head dimension from
//            shared-memory float4 reads (conflict-free: padded rows, and the
//            four query groups of a warp on consecutive rows);
//            the 8 threads of a query group reduce each row's maximum and
//            sum with three shuffles and write P (transposed) and the rescale
//            factor to shared memory;
//   P V:     thread t holds an 8 x (D/16) block of O (queries 8(t/16) + r,
//            dims 4(t%16) + 64c), rescales it and adds the tile's P V.
// The shared-memory pipe bounds this loop (every 16-byte-per-thread load
// costs 4 wavefronts), so the blocks are sized for reuse: 4 FMAs per loaded
// float in P V, 2 in the scores.
// The epilogue divides by the row sums.  When the query tiles are too few to
// fill the GPU (small models), the keys of a tile are split over a cluster of
// up to 8 blocks: each block runs the loop above over its share of the key
// tiles, keeps its unnormalised O and its row maxima and sums in shared
// memory, and after a cluster barrier each block combines a slice of the rows
// from every block's partials through distributed shared memory (no global
// scratch).
#include <math.h>

#include <algorithm>

#include "fademem_internal.h"
#include "per_device.h"

namespace fademem {
namespace {

constexpr int kF32Threads = 128;
constexpr int kBQ = 64;          // queries per block
constexpr int kQS = kBQ / 16;    // score rows per thread: 16 query groups of 8 threads
constexpr int kQO = kBQ / 8;     // output rows per thread: 8 row groups of 16 threads
constexpr int kBK = 32;          // keys per tile
constexpr int kPLD = kBQ + 4;    // row stride of the transposed P tile (floats)

template <int D>
struct F32Smem {
  static constexpr int LD = D + 4;                     // padded row stride of Q and K (floats)
  static constexpr int kQ = 0;                         // [kBQ][LD]
  static constexpr int kK = kQ + kBQ * LD;             // [2][kBK][LD]
  static constexpr int kV = kK + 2 * kBK * LD;         // [2][kBK][D]
  static constexpr int kP = kV + 2 * kBK * D;          // [kBK][kPLD]: P transposed
  static constexpr int kA = kP + kBK * kPLD;           // [kBQ]: rescale factor, then row sums
  static constexpr int kFloats = kA + kBQ;
  static constexpr size_t kBytes = (size_t)kFloats * 4;
};

// 16-byte global -> shared copy that bypasses registers (zero fill if !valid;
// src must still be a valid address).
__device__ __forceinline__ void cp_async16(float* dst, const float* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(valid ? 16 : 0) : "memory");
}

__device__ __forceinline__ float dot4(const float4& a, const float4& b, float acc) {
  acc = fmaf(a.x, b.x, acc);
  acc = fmaf(a.y, b.y, acc);
  acc = fmaf(a.z, b.z, acc);
  return fmaf(a.w, b.w, acc);
}

// Keys: the Lk memory tokens of head h ([Lk][D] at Kc + h * head_stride), then
// the Lk2 current-chunk tokens ([Lk2][H][D] at Kcur).
template <int D>
__global__ void __launch_bounds__(kF32Threads) attend_f32_kernel(
    const float* __restrict__ Kc, const float* __restrict__ Vc, int Lk, const float* __restrict__ Kcur,
    const float* __restrict__ Vcur, int Lk2, const float* __restrict__ Q, float* __restrict__ out, int Lq, int H,
    size_t head_stride, float scale_log2, int csplit, unsigned int* status) {
  using S = F32Smem<D>;
  constexpr int LD = S::LD;
  constexpr int NC = D / 64;  // float4 columns of O per thread and query, 64 dims apart
  extern __shared__ float4 smem4[];
  float* sm = reinterpret_cast<float*>(smem4);
  float* sQ = sm + S::kQ;
  float* sK = sm + S::kK;
  float* sV = sm + S::kV;
  float* sP = sm + S::kP;
  float* sA = sm + S::kA;
  const int t = threadIdx.x;
  // Cluster of csplit blocks (launched with that cluster shape along x): block
  // `rank` of query tile blockIdx.x / csplit takes key tiles [tb, te).
  const int rank = (int)(blockIdx.x % (unsigned)csplit);
  const int q0 = (int)(blockIdx.x / (unsigned)csplit) * kBQ, h = blockIdx.y;
  const int Lt = Lk + Lk2;
  const int n_tiles = (Lt + kBK - 1) / kBK;
  const int kt_begin = (int)((long long)n_tiles * rank / csplit) * kBK;
  const int kt_end = min(Lt, (int)((long long)n_tiles * (rank + 1) / csplit) * kBK);
  // Buffers for the bounds-checking build: the layer's K and V memory, the
  // chunk's K and V, Q and out.
  const DevRange k_r = dev_range(Kc, (size_t)H * head_stride * 4), v_r = dev_range(Vc, (size_t)H * head_stride * 4);
  const DevRange kc_r = dev_range(Kcur, (size_t)Lk2 * H * D * 4), vc_r = dev_range(Vcur, (size_t)Lk2 * H * D * 4);
  const DevRange q_r = dev_range(Q, (size_t)Lq * H * D * 4), o_r = dev_range(out, (size_t)Lq * H * D * 4);

  for (int i = t; i < kBQ * D / 4; i += kF32Threads) {
    const int r = i / (D / 4), c = (i % (D / 4)) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    const float* src = Q + ((size_t)(q0 + r) * H + h) * D + c;
    if (q0 + r < Lq && (!kBoundsChecks || bounds_ok(q_r, src, 16, status))) v = *reinterpret_cast<const float4*>(src);
    *reinterpret_cast<float4*>(sQ + r * LD + c) = v;
  }

  const int qg = t >> 3, kg = t & 7;    // scores: queries qg + 16r; keys kg + 8i
  const int qo = t >> 4, g = t & 15;    // P V: queries kQO qo + r; dims 4g + 64c
  const float* Kh = Kc + (size_t)h * head_stride;  // keys of head h: [Lk][D], slots 0..count-1 contiguous
  const float* Vh = Vc + (size_t)h * head_stride;
  float m_run[kQS], l_run[kQS];
#pragma unroll
  for (int r = 0; r < kQS; ++r) {
    m_run[r] = -INFINITY;
    l_run[r] = 0.f;
  }
  float o[kQO][4 * NC];
#pragma unroll
  for (int r = 0; r < kQO; ++r)
#pragma unroll
    for (int e = 0; e < 4 * NC; ++e) o[r][e] = 0.f;

  // Stage key tile kt (keys kt .. kt + kBK - 1; past the last key: zeros) into buffer buf.
  auto load_tile = [&](int kt, int buf) {
    float* dK = sK + buf * kBK * LD;
    float* dV = sV + buf * kBK * D;
    for (int i = t; i < kBK * D / 4; i += kF32Threads) {
      const int r = i / (D / 4), c = (i % (D / 4)) * 4;
      const int key = kt + r;
      bool ok = key < Lt;
      const float* kp = Q;  // any valid address for a zero-filled copy
      const float* vp = Q;
      if (ok) {
        kp = key < Lk ? Kh + (size_t)key * D + c : Kcur + ((size_t)(key - Lk) * H + h) * D + c;
        vp = key < Lk ? Vh + (size_t)key * D + c : Vcur + ((size_t)(key - Lk) * H + h) * D + c;
        if (kBoundsChecks && !(bounds_ok(key < Lk ? k_r : kc_r, kp, 16, status) &&
                               bounds_ok(key < Lk ? v_r : vc_r, vp, 16, status))) {
          ok = false;
          kp = vp = Q;
        }
      }
      cp_async16(dK + r * LD + c, kp, ok);
      cp_async16(dV + r * D + c, vp, ok);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  if (kt_begin < kt_end) load_tile(kt_begin, 0);
  for (int kt = kt_begin, it = 0; kt < kt_end; kt += kBK, ++it) {
    // Every thread finished reading the other buffer (and P) in the previous
    // iteration, so the next tile may load into it while this one is used.
    if (kt + kBK < kt_end) {
      load_tile(kt + kBK, (it + 1) & 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();  // this tile's copies (every thread's) have landed
    const float* tK = sK + (it & 1) * kBK * LD;
    const float* tV = sV + (it & 1) * kBK * D;

    // ---- scores and the online softmax of rows qg + 16r ----
    float s[kQS][4];
#pragma unroll
    for (int r = 0; r < kQS; ++r)
#pragma unroll
      for (int i = 0; i < 4; ++i) s[r][i] = 0.f;
#pragma unroll 2
    for (int d = 0; d < D; d += 4) {
      float4 q[kQS], k[4];
#pragma unroll
      for (int r = 0; r < kQS; ++r) q[r] = *reinterpret_cast<const float4*>(sQ + (qg + 16 * r) * LD + d);
#pragma unroll
      for (int i = 0; i < 4; ++i) k[i] = *reinterpret_cast<const float4*>(tK + (kg + 8 * i) * LD + d);
#pragma unroll
      for (int r = 0; r < kQS; ++r)
#pragma unroll
        for (int i = 0; i < 4; ++i) s[r][i] = dot4(q[r], k[i], s[r][i]);
    }
#pragma unroll
    for (int r = 0; r < kQS; ++r) {
      float mx = -INFINITY;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        s[r][i] = kt + kg + 8 * i < Lt ? s[r][i] * scale_log2 : -INFINITY;
        mx = fmaxf(mx, s[r][i]);
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      const float m_new = fmaxf(m_run[r], mx);  // finite: every tile holds a key
      const float alpha = exp2f(m_run[r] - m_new);
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float p = exp2f(s[r][i] - m_new);
        sum += p;
        sP[(kg + 8 * i) * kPLD + qg + 16 * r] = p;
      }
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      sum += __shfl_xor_sync(0xffffffffu, sum, 4);
      l_run[r] = l_run[r] * alpha + sum;
      m_run[r] = m_new;
      if (kg == 0) sA[qg + 16 * r] = alpha;
    }
    __syncthreads();

    // ---- O <- alpha O + P V for rows kQO qo .. kQO qo + kQO - 1 ----
    float alr[kQO];
#pragma unroll
    for (int r = 0; r < kQO; r += 4) {
      const float4 al = *reinterpret_cast<const float4*>(sA + kQO * qo + r);
      alr[r] = al.x;
      alr[r + 1] = al.y;
      alr[r + 2] = al.z;
      alr[r + 3] = al.w;
    }
#pragma unroll
    for (int r = 0; r < kQO; ++r)
#pragma unroll
      for (int e = 0; e < 4 * NC; ++e) o[r][e] *= alr[r];
#pragma unroll 2
    for (int k = 0; k < kBK; ++k) {
      float pr[kQO];
#pragma unroll
      for (int r = 0; r < kQO; r += 4) {
        const float4 p4 = *reinterpret_cast<const float4*>(sP + k * kPLD + kQO * qo + r);
        pr[r] = p4.x;
        pr[r + 1] = p4.y;
        pr[r + 2] = p4.z;
        pr[r + 3] = p4.w;
      }
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const float4 v = *reinterpret_cast<const float4*>(tV + k * D + 64 * c + 4 * g);
#pragma unroll
        for (int r = 0; r < kQO; ++r) {
          o[r][4 * c + 0] = fmaf(pr[r], v.x, o[r][4 * c + 0]);
          o[r][4 * c + 1] = fmaf(pr[r], v.y, o[r][4 * c + 1]);
          o[r][4 * c + 2] = fmaf(pr[r], v.z, o[r][4 * c + 2]);
          o[r][4 * c + 3] = fmaf(pr[r], v.w, o[r][4 * c + 3]);
        }
      }
    }
    __syncthreads();  // P, the rescale factors and this buffer are free again
  }

  if (csplit == 1) {
    if (kg == 0) {
#pragma unroll
      for (int r = 0; r < kQS; ++r) sA[qg + 16 * r] = l_run[r];
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kQO; ++r) {
      const int q = q0 + kQO * qo + r;
      if (q >= Lq) continue;
      const float inv = 1.f / sA[kQO * qo + r];
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        float* dst = out + ((size_t)q * H + h) * D + 64 * c + 4 * g;
        if (kBoundsChecks && !bounds_ok(o_r, dst, 16, status)) continue;
        *reinterpret_cast<float4*>(dst) =
            make_float4(o[r][4 * c] * inv, o[r][4 * c + 1] * inv, o[r][4 * c + 2] * inv, o[r][4 * c + 3] * inv);
      }
    }
    return;
  }

  // ---- split keys: combine the cluster's partials ----
  // This block's partials: unnormalised O [kBQ][D] over the K buffers, row
  // maxima and sums (exp2 domain, this block's reference) over the P tile.
  float* pO = sK;
  float* pM = sP;
  float* pL = sP + kBQ;
  if (kg == 0) {
#pragma unroll
    for (int r = 0; r < kQS; ++r) {
      pM[qg + 16 * r] = m_run[r];
      pL[qg + 16 * r] = l_run[r];
    }
  }
#pragma unroll
  for (int r = 0; r < kQO; ++r)
#pragma unroll
    for (int c = 0; c < NC; ++c)
      *reinterpret_cast<float4*>(pO + (kQO * qo + r) * D + 64 * c + 4 * g) =
          make_float4(o[r][4 * c], o[r][4 * c + 1], o[r][4 * c + 2], o[r][4 * c + 3]);
  cluster_sync();  // every block's partials are written and visible to the cluster
  // Block `rank` writes rows [rank * rows, (rank + 1) * rows) of the tile:
  // out = sum_b 2^(m_b - M) O_b / sum_b 2^(m_b - M) l_b with M = max_b m_b.
  const int rows = kBQ / csplit;
  for (int i = t; i < rows * D / 4; i += kF32Threads) {
    const int row = rank * rows + i / (D / 4), c = (i % (D / 4)) * 4;
    float M = -INFINITY;
    for (int b = 0; b < csplit; ++b) M = fmaxf(M, ld_cluster(cluster_addr(pM + row, b)));
    float den = 0.f;
    float4 num = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int b = 0; b < csplit; ++b) {
      const float w = exp2f(ld_cluster(cluster_addr(pM + row, b)) - M);  // 0 for a block with no keys
      den = fmaf(w, ld_cluster(cluster_addr(pL + row, b)), den);
      const float4 ob = ld_cluster4(cluster_addr(pO + row * D + c, b));
      num.x = fmaf(w, ob.x, num.x);
      num.y = fmaf(w, ob.y, num.y);
      num.z = fmaf(w, ob.z, num.z);
      num.w = fmaf(w, ob.w, num.w);
    }
    const int q = q0 + row;
    if (q >= Lq) continue;
    float* dst = out + ((size_t)q * H + h) * D + c;
    if (kBoundsChecks && !bounds_ok(o_r, dst, 16, status)) continue;
    const float inv = 1.f / den;
    *reinterpret_cast<float4*>(dst) = make_float4(num.x * inv, num.y * inv, num.z * inv, num.w * inv);
  }
  cluster_sync();  // no block leaves while another still reads its shared memory
}

template <int D>
cudaError_t launch_f32(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur, const void* Vcur,
                       int Lk2, const float* Q, float* out, int Lq, float scale_log2, unsigned int* status,
                       cudaStream_t stream) {
  constexpr size_t smem = F32Smem<D>::kBytes;
  if (smem > 48 * 1024) {
    // The shared-memory opt-in is a per-device setting: once per device, with it current.
    static PerDevice<char> opt_in;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    char done = 0;
    if (!opt_in.get(dev, [&e](int, char* v) {
          e = cudaFuncSetAttribute(attend_f32_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
          *v = 1;
          return e == cudaSuccess;
        }, &done))
      return e != cudaSuccess ? e : cudaErrorInvalidDevice;
  }
  // Split the keys over a cluster of csplit blocks while the grid is far from
  // filling the GPU (one wave at the kernel's occupancy) and each block keeps
  // at least two key tiles.
  const long long tiles_q = (Lq + kBQ - 1) / kBQ;
  const long long blocks = tiles_q * g.H;
  const int n_tiles = (Lk + Lk2 + kBK - 1) / kBK;
  // Resident blocks per SM by shared memory (each block also reserves 1 KB).
  const long long per_sm = std::max(1, std::min(8, (int)(233472 / (smem + 1024))));
  const long long wave = (long long)current_device_sm_count(148) * per_sm;
  int csplit = 1;
  while (csplit < 8 && blocks * csplit * 2 <= wave && n_tiles >= 4 * csplit) csplit *= 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(tiles_q * csplit), (unsigned)g.H);
  cfg.blockDim = dim3(kF32Threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)csplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, attend_f32_kernel<D>, (const float*)Kc, (const float*)Vc, Lk, (const float*)Kcur,
                            (const float*)Vcur, Lk2, Q, out, Lq, g.H, (size_t)g.M * g.N * g.D, scale_log2, csplit,
                            status);
}

}  // namespace

cudaError_t launch_attend_f32(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur,
                              const void* Vcur, int Lk2, const float* Q, float* out, int Lq, float scale,
                              unsigned int* status, cudaStream_t stream) {
  const float scale_log2 = scale * 1.4426950408889634f;
  if (g.D == 128) return launch_f32<128>(g, Kc, Vc, Lk, Kcur, Vcur, Lk2, Q, out, Lq, scale_log2, status, stream);
  return launch_f32<64>(g, Kc, Vc, Lk, Kcur, Vcur, Lk2, Q, out, Lq, scale_log2, status, stream);
}

}  // namespace fademem
