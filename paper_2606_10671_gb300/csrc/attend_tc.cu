// bf16 attention of the segment's queries over the consolidated memory
// (Sec. 3.3 last paragraph; Sec. 4.1: every denoising step), on the sm_103a
// tensor cores: per head, out = softmax(scale * Q K^T) V over all count*N
// cached keys.
//
// One CTA computes one 128-query tile of one head:
//   warp 4      TMA producer: Q tile once, then K/V tiles of 128 keys into a
//               2-stage ring (128-byte swizzle, zero fill past the last key)
//   warp 5      allocates 512 TMEM columns and issues tcgen05.mma:
//               S_j = Q K_j^T into TMEM buffer j%2 (fp32), and after the
//               softmax of tile j, O += P_j V_j into the TMEM accumulator
//   warps 0-3   softmax, one thread per query row (= TMEM lane): load S_j,
//               online softmax in the exp2 domain with a lazily updated
//               reference maximum (O is rescaled only when the row maximum
//               grows by more than 2^8), write P_j as bf16 into shared memory
//               in the swizzled K-major layout, then the epilogue O / l.
// S_{j+1} is computed while the softmax of tile j runs.  Every mbarrier wait
// is bounded; on time-out the CTA records it in the status word and leaves.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdio.h>

#include "fademem_internal.h"

namespace fademem {
namespace {

constexpr int kBM = 128;        // query rows per tile (TMEM lanes)
constexpr int kBN = 128;        // keys per tile
constexpr int kHD = 128;        // head dimension
constexpr int kStages = 2;
constexpr int kThreads = 192;
constexpr uint32_t kHalfBytes = kBM * 64 * 2;   // 128 rows x 64 bf16 (one swizzle-128B panel)
constexpr uint32_t kTileBytes = 2 * kHalfBytes; // 128 rows x 128 bf16
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTileBytes;
constexpr uint32_t kOffV = kOffK + kStages * kTileBytes;
constexpr uint32_t kOffP = kOffV + kStages * kTileBytes;
constexpr uint32_t kOffBar = kOffP + kTileBytes;
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;  // barriers + alignment slack
constexpr uint32_t kTmemCols = 512;
constexpr long long kWaitLimitCycles = 4000000000LL;  // ~2 s at 2 GHz

// Barrier indices (8 bytes each at kOffBar).
enum { BAR_Q = 0, BAR_KFULL = 1, BAR_VFULL = 3, BAR_KEMPTY = 5, BAR_VEMPTY = 7, BAR_SFULL = 9, BAR_PFULL = 11,
       BAR_ODONE = 12, BAR_FINAL = 13, BAR_COUNT = 14 };

struct AttnParams {
  CUtensorMap tmQ;   // [Lq][H][D]  dims (D, H, Lq), box (64, 1, 128)
  CUtensorMap tmK;   // [H][Lk][D]  dims (D, Lk, H), box (64, 128, 1)
  CUtensorMap tmV;
  __nv_bfloat16* out;
  int Lq, Lk, H;
  float scale_log2;
  unsigned int* status;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait: false on time-out or when another role of the CTA aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > kWaitLimitCycles) return false;
  }
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int c0, int c1,
                                            int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

#define FM_R8(i) "=r"(r[i]), "=r"(r[i + 1]), "=r"(r[i + 2]), "=r"(r[i + 3]), "=r"(r[i + 4]), "=r"(r[i + 5]), \
                 "=r"(r[i + 6]), "=r"(r[i + 7])
#define FM_W8(i) "r"(r[i]), "r"(r[i + 1]), "r"(r[i + 2]), "r"(r[i + 3]), "r"(r[i + 4]), "r"(r[i + 5]), \
                 "r"(r[i + 6]), "r"(r[i + 7])

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : FM_R8(0), FM_R8(8), FM_R8(16), FM_R8(24)
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      FM_W8(0), FM_W8(8), FM_W8(16), FM_W8(24)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor, 128-byte swizzle (tcgen05 format: start,
// leading/stride byte offsets in 16-byte units, version 1 at bit 46, layout 2 at bit 61).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B, A K-major,
// B K-major (b_mn = 0) or MN-major (b_mn = 1), shape M x N.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)b_mn << 16) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&b);
}

__global__ void __launch_bounds__(kThreads, 1) attend_tc_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + kOffBar;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q0 = blockIdx.x * kBM;
  const int h = blockIdx.y;
  const int n_tiles = (p.Lk + kBN - 1) / kBN;

  if (threadIdx.x == 0) {
    s_abort = 0;
    mbar_init(bar(BAR_Q), 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(BAR_KFULL + s), 1);
      mbar_init(bar(BAR_VFULL + s), 1);
      mbar_init(bar(BAR_KEMPTY + s), 1);
      mbar_init(bar(BAR_VEMPTY + s), 1);
      mbar_init(bar(BAR_SFULL + s), 1);
    }
    mbar_init(bar(BAR_PFULL), 128);
    mbar_init(bar(BAR_ODONE), 1);
    mbar_init(bar(BAR_FINAL), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 5) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (warp == 4 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmV)) : "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int* abort_flag = &s_abort;
  auto fail = [&]() {
    *abort_flag = 1;
    atomicOr(p.status, kStatusTimeout);
  };

  if (warp == 4) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint32_t sQ = sbase + kOffQ;
      mbar_expect_tx(bar(BAR_Q), kTileBytes);
      tma_load_3d(sQ, &p.tmQ, bar(BAR_Q), 0, h, q0);
      tma_load_3d(sQ + kHalfBytes, &p.tmQ, bar(BAR_Q), 64, h, q0);
      for (int j = 0; j < n_tiles; ++j) {
        const int s = j % kStages;
        const uint32_t par = ((j / kStages) & 1) ^ 1;
        if (j >= kStages && !mbar_wait(bar(BAR_KEMPTY + s), par, abort_flag)) { fail(); break; }
        const uint32_t sK = sbase + kOffK + s * kTileBytes;
        mbar_expect_tx(bar(BAR_KFULL + s), kTileBytes);
        tma_load_3d(sK, &p.tmK, bar(BAR_KFULL + s), 0, j * kBN, h);
        tma_load_3d(sK + kHalfBytes, &p.tmK, bar(BAR_KFULL + s), 64, j * kBN, h);
        if (j >= kStages && !mbar_wait(bar(BAR_VEMPTY + s), par, abort_flag)) { fail(); break; }
        const uint32_t sV = sbase + kOffV + s * kTileBytes;
        mbar_expect_tx(bar(BAR_VFULL + s), kTileBytes);
        tma_load_3d(sV, &p.tmV, bar(BAR_VFULL + s), 0, j * kBN, h);
        tma_load_3d(sV + kHalfBytes, &p.tmV, bar(BAR_VFULL + s), 64, j * kBN, h);
      }
    }
  } else if (warp == 5) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc_qk = make_idesc(kBM, kBN, 0);
      constexpr uint32_t idesc_pv = make_idesc(kBM, kHD, 1);
      const uint32_t sQ = sbase + kOffQ, sP = sbase + kOffP;
      const uint32_t tO = tmem + 256;
      bool ok = mbar_wait(bar(BAR_Q), 0, abort_flag);
      if (!ok) fail();
      tc_fence_after();
      for (int j = 0; ok && j <= n_tiles; ++j) {
        if (j < n_tiles) {
          const int s = j % kStages;
          if (!mbar_wait(bar(BAR_KFULL + s), (j / kStages) & 1, abort_flag)) { fail(); break; }
          tc_fence_after();
          const uint32_t sK = sbase + kOffK + s * kTileBytes;
          const uint32_t tS = tmem + (j & 1) * 128;
#pragma unroll
          for (int kk = 0; kk < kHD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
            umma_bf16(tS, sw128_desc(sQ + off, 16, 1024), sw128_desc(sK + off, 16, 1024), idesc_qk, kk > 0);
          }
          umma_commit(bar(BAR_SFULL + (j & 1)));
          umma_commit(bar(BAR_KEMPTY + s));
        }
        if (j >= 1) {
          const int jj = j - 1;
          const int s = jj % kStages;
          if (!mbar_wait(bar(BAR_PFULL), jj & 1, abort_flag)) { fail(); break; }
          if (!mbar_wait(bar(BAR_VFULL + s), (jj / kStages) & 1, abort_flag)) { fail(); break; }
          tc_fence_after();
          const uint32_t sV = sbase + kOffV + s * kTileBytes;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk) {
            const uint32_t offp = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
            umma_bf16(tO, sw128_desc(sP + offp, 16, 1024), sw128_desc(sV + kk * 2048, kHalfBytes, 1024), idesc_pv,
                      (jj > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(bar(BAR_ODONE));
          umma_commit(bar(BAR_VEMPTY + s));
        }
      }
      // Drain: every MMA issued above has completed once this barrier flips.
      umma_commit(bar(BAR_FINAL));
      if (!mbar_wait(bar(BAR_FINAL), 0, abort_flag) && !*abort_flag) fail();
    }
  } else {
    // ---------------- softmax + epilogue (warps 0-3, one query row per thread) ----------------
    const int row = warp * 32 + lane;
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    const uint32_t tO = tmem + 256 + lane_off;
    uint8_t* sP = smem + kOffP;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < n_tiles; ++j) {
      if (!mbar_wait(bar(BAR_SFULL + (j & 1)), (j >> 1) & 1, abort_flag)) { fail(); ok = false; break; }
      tc_fence_after();
      float sv[kBN];
      {
        const uint32_t tS = tmem + (j & 1) * 128 + lane_off;
#pragma unroll
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tS + c * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) sv[c * 32 + i] = __uint_as_float(r[i]);
        }
      }
      if (j == n_tiles - 1) {
        const int valid = p.Lk - j * kBN;
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (c >= valid) sv[c] = -INFINITY;
      }
      float mt = sv[0];
#pragma unroll
      for (int c = 1; c < kBN; ++c) mt = fmaxf(mt, sv[c]);
      mt *= p.scale_log2;
      // Lazy reference maximum: move it only when the tile exceeds it by > 8 (2^8 headroom).
      const bool move = (m_run == -INFINITY) || (mt > m_run + 8.0f);
      const float m_new = move ? fmaxf(mt, m_run) : m_run;
      const float alpha = ex2(m_run - m_new);  // 0 on the first tile, 1 if unchanged
      float rs = 0.f;
      uint32_t pk[kBN / 2];
#pragma unroll
      for (int c = 0; c < kBN; c += 2) {
        const float e0 = ex2(fmaf(sv[c], p.scale_log2, -m_new));
        const float e1 = ex2(fmaf(sv[c + 1], p.scale_log2, -m_new));
        rs += e0 + e1;
        pk[c / 2] = pack_bf16(e0, e1);
      }
      l_run = l_run * alpha + rs;
      m_run = m_new;
      if (j > 0) {
        // PV of tile j-1 must be done: P is overwritten and O may be rescaled.
        if (!mbar_wait(bar(BAR_ODONE), (j - 1) & 1, abort_flag)) { fail(); ok = false; break; }
        tc_fence_after();
        if (__any_sync(0xffffffffu, move)) {
#pragma unroll
          for (int c = 0; c < kHD / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(tO + c * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
            tmem_st32(tO + c * 32, r);
          }
          tmem_st_wait();
        }
      }
      // P row -> shared memory, K-major with 128-byte swizzle (16-byte chunk c of
      // row r lands at chunk c ^ (r % 8) of that row's 128-byte line).
#pragma unroll
      for (int c = 0; c < kBN / 8; ++c) {
        const uint32_t off = (c >> 3) * kHalfBytes + row * 128 + ((((c & 7) ^ (row & 7))) << 4);
        *reinterpret_cast<uint4*>(sP + off) = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      mbar_arrive(bar(BAR_PFULL));
    }
    if (ok && n_tiles > 0) {
      if (!mbar_wait(bar(BAR_ODONE), (n_tiles - 1) & 1, abort_flag)) {
        fail();
      } else {
        tc_fence_after();
        const float inv = 1.f / l_run;
        const int q = q0 + row;
        __nv_bfloat16* orow = p.out + ((size_t)q * p.H + h) * kHD;
#pragma unroll
        for (int c = 0; c < kHD / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tO + c * 32, r);
          tmem_ld_wait();
          if (q < p.Lq) {
#pragma unroll
            for (int i = 0; i < 32; i += 8) {
              uint4 v;
              v.x = pack_bf16(__uint_as_float(r[i]) * inv, __uint_as_float(r[i + 1]) * inv);
              v.y = pack_bf16(__uint_as_float(r[i + 2]) * inv, __uint_as_float(r[i + 3]) * inv);
              v.z = pack_bf16(__uint_as_float(r[i + 4]) * inv, __uint_as_float(r[i + 5]) * inv);
              v.w = pack_bf16(__uint_as_float(r[i + 6]) * inv, __uint_as_float(r[i + 7]) * inv);
              *reinterpret_cast<uint4*>(orow + c * 32 + i) = v;
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

bool encode_3d(EncodeTiledFn enc, CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
               uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2) {
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {b0, b1, b2};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_attend_bf16(const Geometry& g, const void* Kc, const void* Vc, const void* Q, void* out, int Lq,
                               int Lk, float scale, unsigned int* status, cudaStream_t stream, char* err,
                               size_t errlen) {
  if (g.D != kHD) {
    snprintf(err, errlen, "bf16 attention supports head_dim 128 only (got %d)", g.D);
    return cudaErrorNotSupported;
  }
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) {
    snprintf(err, errlen, "cuTensorMapEncodeTiled is unavailable from the driver");
    return cudaErrorNotSupported;
  }
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attend_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  AttnParams prm;
  const uint64_t row = (uint64_t)kHD * 2;
  if (!encode_3d(enc, &prm.tmQ, Q, kHD, g.H, Lq, row, row * g.H, 64, 1, kBM) ||
      !encode_3d(enc, &prm.tmK, Kc, kHD, Lk, g.H, row, row * g.M * g.N, 64, kBN, 1) ||
      !encode_3d(enc, &prm.tmV, Vc, kHD, Lk, g.H, row, row * g.M * g.N, 64, kBN, 1)) {
    snprintf(err, errlen, "cuTensorMapEncodeTiled rejected a tensor map (Lq=%d Lk=%d)", Lq, Lk);
    return cudaErrorInvalidValue;
  }
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.Lq = Lq;
  prm.Lk = Lk;
  prm.H = g.H;
  prm.scale_log2 = scale * 1.4426950408889634f;
  prm.status = status;
  dim3 grid((Lq + kBM - 1) / kBM, g.H);
  attend_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(prm);
  return cudaGetLastError();
}

}  // namespace fademem
