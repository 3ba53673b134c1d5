// fp32 attention of query tokens over the memory (Sec. 3.3 last paragraph:
// the memory is the cached context the backbone's attention sees).
// Exact-precision path for the fp32 storage dtype: one warp per (query, head),
// lanes split the head dimension, online softmax over every cached key in
// fp32 (tf32 tensor cores would not meet a 1e-5 relative tolerance).
#include <math.h>

#include "fademem_internal.h"

namespace fademem {
namespace {

// Keys: the Lk memory tokens of head h ([Lk][D] at Kc + h * head_stride), then
// the Lk2 current-chunk tokens ([Lk2][H][D] at Kcur).
template <int D>
__global__ void __launch_bounds__(256) attend_f32_kernel(const float* __restrict__ Kc, const float* __restrict__ Vc,
                                                         int Lk, const float* __restrict__ Kcur,
                                                         const float* __restrict__ Vcur, int Lk2,
                                                         const float* __restrict__ Q, float* __restrict__ out,
                                                         int Lq, int H, size_t head_stride, float scale_log2,
                                                         unsigned int* status) {
  constexpr int P = D / 32;
  const int lane = threadIdx.x & 31;
  const long long gw = (long long)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (gw >= (long long)Lq * H) return;
  const int q = (int)(gw / H), h = (int)(gw % H);
  const float* qp = Q + ((size_t)q * H + h) * D;
  // Buffers for the bounds-checking build: the layer's K and V memory, the
  // chunk's K and V, Q and out.
  const DevRange k_r = dev_range(Kc, (size_t)H * head_stride * 4), v_r = dev_range(Vc, (size_t)H * head_stride * 4);
  const DevRange kc_r = dev_range(Kcur, (size_t)Lk2 * H * D * 4), vc_r = dev_range(Vcur, (size_t)Lk2 * H * D * 4);
  const DevRange q_r = dev_range(Q, (size_t)Lq * H * D * 4), o_r = dev_range(out, (size_t)Lq * H * D * 4);
  if (kBoundsChecks && !bounds_ok(q_r, qp, D * 4, status)) return;
  float qv[P], o[P];
#pragma unroll
  for (int i = 0; i < P; ++i) { qv[i] = qp[lane + 32 * i]; o[i] = 0.f; }
  const float* Kh = Kc + (size_t)h * head_stride;  // keys of head h: [Lk][D], slots 0..count-1 contiguous
  const float* Vh = Vc + (size_t)h * head_stride;
  float m = -INFINITY, l = 0.f;
  for (int k = 0; k < Lk + Lk2; ++k) {
    const float* kr = k < Lk ? Kh + (size_t)k * D : Kcur + ((size_t)(k - Lk) * H + h) * D;
    const float* vr = k < Lk ? Vh + (size_t)k * D : Vcur + ((size_t)(k - Lk) * H + h) * D;
    if (kBoundsChecks &&
        (!bounds_ok(k < Lk ? k_r : kc_r, kr, D * 4, status) || !bounds_ok(k < Lk ? v_r : vc_r, vr, D * 4, status)))
      continue;
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < P; ++i) dot = fmaf(qv[i], kr[lane + 32 * i], dot);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    const float s = dot * scale_log2;
    const float m_new = fmaxf(m, s);
    const float c = exp2f(m - m_new);
    const float p = exp2f(s - m_new);
    l = l * c + p;
#pragma unroll
    for (int i = 0; i < P; ++i) o[i] = fmaf(p, vr[lane + 32 * i], o[i] * c);
    m = m_new;
  }
  float* op = out + ((size_t)q * H + h) * D;
  if (kBoundsChecks && !bounds_ok(o_r, op, D * 4, status)) return;
  const float inv = 1.f / l;
#pragma unroll
  for (int i = 0; i < P; ++i) op[lane + 32 * i] = o[i] * inv;
}

}  // namespace

cudaError_t launch_attend_f32(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur,
                              const void* Vcur, int Lk2, const float* Q, float* out, int Lq, float scale,
                              unsigned int* status, cudaStream_t stream) {
  const long long warps = (long long)Lq * g.H;
  const int threads = 256;
  const long long blocks = (warps * 32 + threads - 1) / threads;
  const float scale_log2 = scale * 1.4426950408889634f;
  const size_t head_stride = (size_t)g.M * g.N * g.D;
  if (g.D == 128)
    attend_f32_kernel<128><<<(unsigned)blocks, threads, 0, stream>>>(
        (const float*)Kc, (const float*)Vc, Lk, (const float*)Kcur, (const float*)Vcur, Lk2, Q, out, Lq, g.H,
        head_stride, scale_log2, status);
  else
    attend_f32_kernel<64><<<(unsigned)blocks, threads, 0, stream>>>(
        (const float*)Kc, (const float*)Vc, Lk, (const float*)Kcur, (const float*)Vcur, Lk2, Q, out, Lq, g.H,
        head_stride, scale_log2, status);
  return cudaGetLastError();
}

}  // namespace fademem
