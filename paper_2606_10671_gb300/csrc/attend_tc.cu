// bf16 attention of the segment's queries over the consolidated memory
// (Sec. 3.3 last paragraph; Sec. 4.1: every denoising step), on the sm_103a
// tensor cores: per head, out = softmax(scale * Q K^T) V over all count*N
// cached keys.
//
// One CTA computes one 128-query tile of one head, 352 threads:
//   warp 8      TMA producer of Q (once) and of K tiles of 128 keys into a
//               3-stage ring (128-byte swizzle, zero fill past the last key)
//   warp 10     TMA producer of V tiles into a 3-stage ring, so a slow V slot
//               never holds back the next K tile
//   warp 9      allocates 512 TMEM columns and issues tcgen05.mma
//   warps 0-7   two softmax groups of four warps; group g takes the key tiles
//               j = g, g+2, ... with its own online-softmax state (m, l) and
//               its own accumulator O_g in TMEM (one query row per thread =
//               TMEM lane).  Per tile: load S_j, exp2-domain softmax with a
//               lazily updated reference maximum (O_g is rescaled only when
//               the row maximum grows by more than 2^8), write P_j as bf16
//               pairs over S_j in TMEM.
// P_j V_j reads P from TMEM (tcgen05.mma with the A operand in TMEM), so the
// only shared-memory traffic per tile is Q and the K/V tiles.  While one group
// runs its softmax, the tensor pipe runs the other group's P·V and next Q·K^T,
// so the tensor pipe and the exponential unit overlap.  The epilogue combines
// (O_0, m_0, l_0) and (O_1, m_1, l_1) row by row.  Every mbarrier wait is
// bounded; on time-out the CTA records it in the status word and leaves.
//
// When the tiles are too few to fill half the SMs, a tile's key tiles are
// split over a thread-block cluster of 2, 4 or 8 CTAs (attend_tc_kernel<true>),
// each running the pipeline above over its share and leaving its unnormalised
// (O, m, l) in shared memory; after a cluster barrier each CTA assembles a
// slice of the tile's rows from all of them through distributed shared memory.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdio.h>

#include "fademem_internal.h"
#include "per_device.h"

namespace fademem {
namespace {

constexpr int kBM = 128;        // query rows per tile (TMEM lanes)
constexpr int kBN = 128;        // keys per tile
constexpr int kHD = 128;        // head dimension
constexpr int kSoftmaxThreads = 256;  // two groups of four warps
constexpr int kWarpTma = 8;    // Q and K producer
constexpr int kWarpMma = 9;
constexpr int kWarpTmaV = 10;  // V producer
constexpr int kThreads = 352;
constexpr int kKStages = 3;
constexpr int kVStages = 3;
constexpr uint32_t kHalfBytes = kBM * 64 * 2;   // 128 rows x 64 bf16 (one swizzle-128B panel)
constexpr uint32_t kTileBytes = 2 * kHalfBytes; // 128 rows x 128 bf16
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTileBytes;
constexpr uint32_t kOffV = kOffK + kKStages * kTileBytes;
constexpr uint32_t kOffBar = kOffV + kVStages * kTileBytes;
// Per-row (m, l) of both groups for the epilogue: reuses K stage 0, which no
// MMA reads any more once the final drain has completed.
constexpr uint32_t kOffML = kOffK;
// Row stride (floats) of a split tile's partial O in shared memory: 4 floats of
// padding keep the rows' 16-byte stores and loads on distinct banks.
constexpr int kPOStride = kHD + 4;
static_assert((kBM * kPOStride + 2 * kBM) * 4 <= kVStages * kTileBytes, "split partials fit the V ring");
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;  // + alignment slack
constexpr uint32_t kTmemCols = 512;
// TMEM columns: S_0 [0,128), S_1 [128,256) fp32 (P_g overwrites the first 64
// columns of S_g as bf16 pairs); O_0 [256,384), O_1 [384,512) fp32.
constexpr uint32_t kColO = 256;
constexpr long long kWaitLimitCycles = 4000000000LL;  // ~2 s at 2 GHz

// Barrier indices (8 bytes each at kOffBar).
enum { BAR_Q = 0, BAR_KFULL = 1, BAR_KEMPTY = 4, BAR_VFULL = 7, BAR_VEMPTY = 10, BAR_SFULL = 13, BAR_PFULL = 15,
       BAR_FINAL = 17, BAR_COUNT = 18 };

struct AttnParams {
  CUtensorMap tmQ;   // [Lq][H][D]  dims (D, H, Lq), box (64, 1, 128)
  CUtensorMap tmK;   // memory keys [H][Lk][D]  dims (D, Lk, H), box (64, 128, 1)
  CUtensorMap tmV;
  CUtensorMap tmK2;  // current-chunk keys [Lk2][H][D]  dims (D, H, Lk2), box (64, 1, 128)
  CUtensorMap tmV2;
  __nv_bfloat16* out;
  int Lq, Lk, Lk2, H;
  int csplit;  // CTAs (a cluster) sharing one query tile's key tiles: 1, 2, 4 or 8
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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          long long limit = kWaitLimitCycles) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) return false;
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
// Same, with the A operand in TMEM (rows on lanes, two 16-bit elements per column).
__device__ __forceinline__ void umma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
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
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16};" ::"r"(taddr),
      FM_W8(0), FM_W8(8)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// Wait for this thread's outstanding TMEM loads, with r as an in/out operand
// so that no use of the loaded registers is scheduled before the wait.
__device__ __forceinline__ void tmem_ld_wait_regs(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
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
// Packed two-lane fp32 arithmetic (one fma.rn.f32x2 / add.rn.f32x2 for two
// values): the softmax is bound by instruction issue, so pairs halve its
// FFMA/FADD count.  The float2 builtins let the compiler place the pairs in
// register pairs itself.
__device__ __forceinline__ void ffma2(float& d0, float& d1, float a0, float a1, float b0, float b1, float c0,
                                      float c1) {
  const float2 d = __ffma2_rn(make_float2(a0, a1), make_float2(b0, b1), make_float2(c0, c1));
  d0 = d.x;
  d1 = d.y;
}
__device__ __forceinline__ void fadd2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
  const float2 d = __fadd2_rn(make_float2(a0, a1), make_float2(b0, b1));
  d0 = d.x;
  d1 = d.y;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&b);
}

// Row-sum bound of the softmax fast path: every exponential of the row is at
// most the sum, so P stays far inside bf16/fp32 range.
constexpr float kFastRowSumLimit = 65536.f;

// Exponentials of one quarter (32 keys, keys 32 qtr .. 32 qtr + 31) of this
// thread's row of S, packed into pk16 (bf16 pairs, the quarter's 16 P columns).
template <bool kRagged>
__device__ __forceinline__ void exp_quarter16(const uint32_t (&r)[32], int qtr, int valid, float scale_log2,
                                              float neg_m, float& rs0, float& rs1, uint32_t (&pk16)[16]) {
#pragma unroll
  for (int c = 0; c < 32; c += 2) {
    float x0, x1;
    ffma2(x0, x1, __uint_as_float(r[c]), __uint_as_float(r[c + 1]), scale_log2, scale_log2, neg_m, neg_m);
    if (kRagged) {
      if (32 * qtr + c >= valid) x0 = -INFINITY;
      if (32 * qtr + c + 1 >= valid) x1 = -INFINITY;
    }
    const float e0 = ex2(x0);
    const float e1 = ex2(x1);
    fadd2(rs0, rs1, rs0, rs1, e0, e1);
    pk16[c / 2] = pack_bf16(e0, e1);
  }
}
__device__ __forceinline__ uint32_t barat(uint32_t bar0, int i) { return bar0 + 8u * (uint32_t)i; }

__device__ __noinline__ void record_timeout(volatile int* abort_flag, unsigned int* status) {
  *abort_flag = 1;
  atomicOr(status, kStatusTimeout);
}

// The 8 MMAs (K = 128 in steps of 16) of S = Q K^T for one key tile, issued
// back to back: every operand is a by-value register and the descriptors only
// advance by constants, so nothing between two tcgen05.mma stalls the issuer.
__device__ __forceinline__ void issue_qk8(uint32_t tS, uint64_t dQ, uint64_t dK, uint32_t idesc) {
#pragma unroll
  for (int kk = 0; kk < kHD / 16; ++kk) {
    const uint64_t off = (uint64_t)(((kk >> 2) * kHalfBytes + (kk & 3) * 32) >> 4);
    umma_bf16(tS, dQ + off, dK + off, idesc, kk > 0 ? 1u : 0u);
  }
}
// The 8 MMAs of O += P V for one key tile (P in TMEM, 16 keys = 8 columns per step).
__device__ __forceinline__ void issue_pv8(uint32_t tO, uint32_t tP, uint64_t dV, uint32_t idesc, uint32_t acc0) {
#pragma unroll
  for (int kk = 0; kk < kBN / 16; ++kk)
    umma_bf16_ts(tO, tP + kk * 8, dV + (uint64_t)(kk * (2048 >> 4)), idesc, kk > 0 ? 1u : acc0);
}

// kSplit: the query tile's keys are split over a cluster of p.csplit CTAs.  The
// whole-tile instance (kSplit = false) keeps none of the split's bookkeeping.
template <bool kSplit>
__global__ void __launch_bounds__(kThreads, 1) attend_tc_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + kOffBar;
  float* s_ml = reinterpret_cast<float*>(smem + kOffML);  // [2 groups][2 (m, l)][128 rows]
  // A split tile's partials for the cluster's combine, over the V ring (idle
  // once every MMA has completed): O [128][kPOStride], then m [128] and l [128].
  float* s_po = reinterpret_cast<float*>(smem + kOffV);
  float* s_pm = s_po + kBM * kPOStride;
  float* s_pl = s_pm + kBM;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // A query tile's key tiles may be split over a cluster of p.csplit CTAs
  // (launched with that cluster shape along x): CTA `rank` takes key tiles
  // [tb, tb + n_tiles) of the n_all, and the cluster combines its partials.
  const int csplit = kSplit ? p.csplit : 1;
  const int rank = kSplit ? (int)(blockIdx.x % (unsigned)csplit) : 0;
  const int q0 = kSplit ? (int)(blockIdx.x / (unsigned)csplit) * kBM : (int)blockIdx.x * kBM;
  const int h = blockIdx.y;
  if (kBoundsChecks && threadIdx.x == 0) index_ok(h, p.H, p.status);
  // Key tiles 0..n1-1 come from the memory, n1..n1+n2-1 from the current chunk.
  const int n1 = (p.Lk + kBN - 1) / kBN;
  const int n_all = n1 + (p.Lk2 + kBN - 1) / kBN;
  const int tb = kSplit ? n_all * rank / csplit : 0;
  const int n_tiles = kSplit ? n_all * (rank + 1) / csplit - tb : n_all;  // this CTA's key tiles (>= 4 when split)
  constexpr bool split = kSplit;

  if (threadIdx.x == 0) {
    s_abort = 0;
    mbar_init(barat(bar0, BAR_Q), 1);
    for (int s = 0; s < kKStages; ++s) {
      mbar_init(barat(bar0, BAR_KFULL + s), 1);
      mbar_init(barat(bar0, BAR_KEMPTY + s), 1);
    }
    for (int s = 0; s < kVStages; ++s) {
      mbar_init(barat(bar0, BAR_VFULL + s), 1);
      mbar_init(barat(bar0, BAR_VEMPTY + s), 1);
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(barat(bar0, BAR_SFULL + g), 1);
      mbar_init(barat(bar0, BAR_PFULL + g), 128);
    }
    mbar_init(barat(bar0, BAR_FINAL), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == kWarpMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (warp == kWarpTma && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmV)) : "memory");
    if (p.Lk2 > 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmK2)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmV2)) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // Launched as a programmatic dependent: the set-up above overlaps the
  // previous kernel; nothing in global memory is touched before this wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const uint32_t tmem = s_tmem;
  volatile int* abort_flag = &s_abort;

  if (warp == kWarpTma) {
    // ---------------- TMA producer of Q (once) and K_j into stage j%3 ----------------
    if (lane == 0) {
      const uint32_t sQ = sbase + kOffQ;
      mbar_expect_tx(barat(bar0, BAR_Q), kTileBytes);
      tma_load_3d(sQ, &p.tmQ, barat(bar0, BAR_Q), 0, h, q0);
      tma_load_3d(sQ + kHalfBytes, &p.tmQ, barat(bar0, BAR_Q), 64, h, q0);
      for (int j = 0; j < n_tiles; ++j) {
        const int s = j % kKStages;
        const uint32_t full = barat(bar0, BAR_KFULL + s);
        if (j >= kKStages && !mbar_wait(barat(bar0, BAR_KEMPTY + s), ((j / kKStages) & 1) ^ 1, abort_flag)) {
          record_timeout(abort_flag, p.status);
          break;
        }
        const uint32_t sK = sbase + kOffK + s * kTileBytes;
        const int t = tb + j;  // key tile
        if (kBoundsChecks && !index_ok(t < n1 ? (long long)t * kBN : (long long)(t - n1) * kBN, t < n1 ? p.Lk : p.Lk2,
                                       p.status)) {
          *abort_flag = 1;  // stop the CTA: every role's waits give up on the abort flag
          break;
        }
        mbar_expect_tx(full, kTileBytes);
        if (t < n1) {
          tma_load_3d(sK, &p.tmK, full, 0, t * kBN, h);
          tma_load_3d(sK + kHalfBytes, &p.tmK, full, 64, t * kBN, h);
        } else {
          tma_load_3d(sK, &p.tmK2, full, 0, h, (t - n1) * kBN);
          tma_load_3d(sK + kHalfBytes, &p.tmK2, full, 64, h, (t - n1) * kBN);
        }
      }
    }
  } else if (warp == kWarpTmaV) {
    // ---------------- TMA producer of V_j into stage j%3 (independent of the K ring) ----------------
    if (lane == 0) {
      for (int j = 0; j < n_tiles; ++j) {
        const int s = j % kVStages;
        const uint32_t full = barat(bar0, BAR_VFULL + s);
        if (j >= kVStages && !mbar_wait(barat(bar0, BAR_VEMPTY + s), ((j / kVStages) & 1) ^ 1, abort_flag)) {
          record_timeout(abort_flag, p.status);
          break;
        }
        const uint32_t sV = sbase + kOffV + s * kTileBytes;
        const int t = tb + j;  // key tile
        mbar_expect_tx(full, kTileBytes);
        if (t < n1) {
          tma_load_3d(sV, &p.tmV, full, 0, t * kBN, h);
          tma_load_3d(sV + kHalfBytes, &p.tmV, full, 64, t * kBN, h);
        } else {
          tma_load_3d(sV, &p.tmV2, full, 0, h, (t - n1) * kBN);
          tma_load_3d(sV + kHalfBytes, &p.tmV2, full, 64, h, (t - n1) * kBN);
        }
      }
    }
  } else if (warp == kWarpMma) {
    // ---------------- MMA issuer ----------------
    // Tile j belongs to softmax group j%2: S_j goes to TMEM buffer j%2, the group
    // writes P_j over the first 64 columns of that buffer, and P_j V_j goes to the
    // group's own accumulator O_{j%2}.  The tensor pipe runs tcgen05.mma in issue
    // order, so issuing S_{j+2} after P_j V_j never overwrites P_j too early.
    // One commit per tile: a commit costs the tensor pipe about as much as an MMA,
    // so K/V slot release is signalled by the softmax groups, not here.
    if (lane == 0) {
      constexpr uint32_t idesc_qk = make_idesc(kBM, kBN, 0);
      constexpr uint32_t idesc_pv = make_idesc(kBM, kHD, 1);
      const uint64_t dQ = sw128_desc(sbase + kOffQ, 16, 1024);
      const uint64_t dK0 = sw128_desc(sbase + kOffK, 16, 1024);
      const uint64_t dV0 = sw128_desc(sbase + kOffV, kHalfBytes, 1024);
      constexpr uint64_t kStageStep = kTileBytes >> 4;  // descriptor advance per 32 KB stage
      bool ok = mbar_wait(barat(bar0, BAR_Q), 0, abort_flag);
      for (int j = 0; ok && j < 2 && j < n_tiles; ++j) {
        const int s = j % kKStages;
        if (!mbar_wait(barat(bar0, BAR_KFULL + s), (j / kKStages) & 1, abort_flag)) { ok = false; break; }
        tc_fence_after();
        issue_qk8(tmem + (j & 1) * kBN, dQ, dK0 + s * kStageStep, idesc_qk);
        umma_commit(barat(bar0, BAR_SFULL + (j & 1)));
      }
      for (int j = 0; ok && j < n_tiles; ++j) {
        const int g = j & 1, sv = j % kVStages;
        // K_{j+2} and V_j (usually loaded long before) are waited for first and
        // P_j, the wait that blocks, last, so that the tile's 16 MMAs go out as
        // one burst with no wait between P_j V_j and Q K_{j+2}^T.  Neither load
        // waits for P_j: their slots are freed by the completion of S_{j-1}
        // (Q K_{j-1}^T, and P_{j-3} V_{j-3} issued before it).
        const int jn = j + 2;
        const int sk = jn % kKStages;
        if ((jn < n_tiles && !mbar_wait(barat(bar0, BAR_KFULL + sk), (jn / kKStages) & 1, abort_flag)) ||
            !mbar_wait(barat(bar0, BAR_VFULL + sv), (j / kVStages) & 1, abort_flag) ||
            !mbar_wait(barat(bar0, BAR_PFULL + g), (j >> 1) & 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        issue_pv8(tmem + kColO + g * kHD, tmem + g * kBN, dV0 + sv * kStageStep, idesc_pv, j >= 2 ? 1u : 0u);
        if (jn < n_tiles) {
          issue_qk8(tmem + g * kBN, dQ, dK0 + sk * kStageStep, idesc_qk);
          // Completes with P_j V_j and S_{j+2}: the group's next S, and (through it)
          // the release of V slot j%3 and K slot (j+2)%3.
          umma_commit(barat(bar0, BAR_SFULL + g));
        }
      }
      if (!ok && !*abort_flag) record_timeout(abort_flag, p.status);
      // Drain: every MMA issued above has completed once this barrier flips.
      umma_commit(barat(bar0, BAR_FINAL));
      if (!mbar_wait(barat(bar0, BAR_FINAL), 0, abort_flag) && !*abort_flag) record_timeout(abort_flag, p.status);
    }
  } else {
    // ---------------- softmax groups 0/1 (warps 0-3 / 4-7), one query row per thread ----------------
    const int grp = warp >> 2;
    const int row = (warp & 3) * 32 + lane;
    const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + grp * kBN + lane_off;
    const uint32_t tO = tmem + kColO + grp * kHD + lane_off;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = grp; j < n_tiles; j += 2) {
      if (!mbar_wait(barat(bar0, BAR_SFULL + grp), (j >> 1) & 1, abort_flag)) { record_timeout(abort_flag, p.status); ok = false; break; }
      if ((threadIdx.x & 127) == 0) {
        // S_j complete means Q K_j^T and (issued before it) P_{j-2} V_{j-2} are done:
        // K slot j%3 and V slot (j-2)%3 may be refilled.
        mbar_arrive(barat(bar0, BAR_KEMPTY + j % kKStages));
        if (j >= 2) mbar_arrive(barat(bar0, BAR_VEMPTY + (j - 2) % kVStages));
      }
      tc_fence_after();
      const int t = tb + j;  // key tile
      const int valid = t < n1 ? p.Lk - t * kBN : p.Lk2 - (t - n1) * kBN;  // keys of this tile
      // Fast path: exponentials against the running reference maximum m_run,
      // with no max over the tile first.  Any reference keeps the softmax exact
      // (it cancels in O / l) as long as no exponential overflows, and the row
      // sum bounds every term of the row, so a sum <= 2^16 (finite, not NaN)
      // proves the tile safe.  The TMEM load of the next quarter of S overlaps
      // the exponentials of the current one.  P is held in registers until the
      // check passes, so S is still intact for the slow path.
      // The whole row of S goes to registers at once (one wait), so P can be
      // written over S in TMEM quarter by quarter as it is computed, and the
      // rare slow path recomputes from the registers.
      uint32_t r[4][32];
      tmem_ld32(tS, r[0]);
      tmem_ld32(tS + 32, r[1]);
      tmem_ld32(tS + 64, r[2]);
      tmem_ld32(tS + 96, r[3]);
      tmem_ld_wait_regs(r[0]);
      tmem_ld_wait_regs(r[1]);
      tmem_ld_wait_regs(r[2]);
      tmem_ld_wait_regs(r[3]);
      if (j < 2) {
        // The group's first tile has no reference yet: take its row maximum.
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (32 * c + i < valid) mx = fmaxf(mx, __uint_as_float(r[c][i]));
        m_run = mx * p.scale_log2;  // finite: every tile holds at least one key
      }
      // Fast path: exponentials against the running reference maximum m_run,
      // with no max over the tile.  Any reference keeps the softmax exact (it
      // cancels in O / l) as long as no exponential overflows, and the row sum
      // bounds every term of the row, so a sum <= 2^16 (finite, not NaN) proves
      // the tile safe.  P quarter q (keys 32q..32q+31) goes to P columns 16q..,
      // which held S columns already in registers.
      float rs0 = 0.f, rs1 = 0.f;
      {
        const float neg_m = -m_run;
#pragma unroll
        for (int qtr = 0; qtr < 4; ++qtr) {
          uint32_t pk16[16];
          if (valid < kBN) exp_quarter16<true>(r[qtr], qtr, valid, p.scale_log2, neg_m, rs0, rs1, pk16);
          else exp_quarter16<false>(r[qtr], qtr, valid, p.scale_log2, neg_m, rs0, rs1, pk16);
          tmem_st16(tS + 16 * qtr, pk16);
        }
      }
      float alpha = 1.f;
      bool moved = false;
      if (__any_sync(0xffffffffu, !(rs0 + rs1 <= kFastRowSumLimit))) {
        // Slow path (a row maximum that outgrew the reference): take the tile
        // maximum from the registers, move the reference lazily (only when the
        // tile exceeds it by more than 2^8) and write P again.
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            const float s0 = 32 * c + i < valid ? __uint_as_float(r[c][i]) : -INFINITY;
            const float s1 = 32 * c + i + 1 < valid ? __uint_as_float(r[c][i + 1]) : -INFINITY;
            mx = fmax3(mx, s0, s1);
          }
        const float mt = mx * p.scale_log2;
        const bool move = mt > m_run + 8.0f;
        const float m_new = move ? fmaxf(mt, m_run) : m_run;
        alpha = ex2(m_run - m_new);  // 1 if unchanged
        m_run = m_new;
        rs0 = 0.f;
        rs1 = 0.f;
        tmem_st_wait();  // the fast path's stores of P land before they are overwritten
#pragma unroll
        for (int qtr = 0; qtr < 4; ++qtr) {
          uint32_t pk16[16];
          exp_quarter16<true>(r[qtr], qtr, valid, p.scale_log2, -m_new, rs0, rs1, pk16);
          tmem_st16(tS + 16 * qtr, pk16);
        }
        moved = __any_sync(0xffffffffu, move);
      }
      l_run = l_run * alpha + (rs0 + rs1);
      if (j >= 2 && moved) {
        // Rescale O_grp before P_j V_j accumulates into it.  Its last update
        // (P_{j-2} V_{j-2}) was issued before S_j, so it is complete once S_j is.
#pragma unroll
        for (int c = 0; c < kHD / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tO + c * 32, r);
          tmem_ld_wait_regs(r);
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
          tmem_st32(tO + c * 32, r);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(barat(bar0, BAR_PFULL + grp));
    }
    // ---------------- epilogue: combine the two groups' (O, m, l) ----------------
    const bool fin = ok && !*abort_flag && mbar_wait(barat(bar0, BAR_FINAL), 0, abort_flag);
    if (ok && !fin) record_timeout(abort_flag, p.status);
    s_ml[(grp * 2 + 0) * kBM + row] = m_run;  // K stage 0 is idle once every MMA has completed
    s_ml[(grp * 2 + 1) * kBM + row] = l_run;
    asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
    if (fin && !*abort_flag) {
      {
        tc_fence_after();
        const float m0 = s_ml[0 * kBM + row], l0 = s_ml[1 * kBM + row];
        const float m1 = s_ml[2 * kBM + row], l1 = s_ml[3 * kBM + row];
        const bool has1 = n_tiles > 1;
        const float m = has1 ? fmaxf(m0, m1) : m0;
        const float f0 = ex2(m0 - m);
        const float f1 = has1 ? ex2(m1 - m) : 0.f;
        const float l = l0 * f0 + l1 * f1;
        // A split tile keeps this CTA's O unnormalised (relative to m) for the
        // cluster's combine; a whole tile is divided by l here.
        const float inv = split ? 1.f : 1.f / l;
        const float a0 = f0 * inv, a1 = f1 * inv;
        const int q = q0 + row;
        if (split && grp == 0) {
          s_pm[row] = m;
          s_pl[row] = l;
        }
        __nv_bfloat16* orow = p.out + ((size_t)q * p.H + h) * kHD;
        const uint32_t tO0 = tmem + kColO + lane_off;
        const uint32_t tO1 = tmem + kColO + kHD + lane_off;
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int col = grp * 64 + c * 32;  // this group writes columns [64 grp, 64 grp + 64)
          uint32_t r0[32], r1[32];
          tmem_ld32(tO0 + col, r0);
          if (has1) tmem_ld32(tO1 + col, r1);
          tmem_ld_wait();
          if (q < p.Lq) {
#pragma unroll
            for (int i = 0; i < 32; i += 8) {
              float o[8];
#pragma unroll
              for (int e = 0; e < 8; ++e)
                o[e] = __uint_as_float(r0[i + e]) * a0 + (has1 ? __uint_as_float(r1[i + e]) * a1 : 0.f);
              if (split) {
                float4* dst = reinterpret_cast<float4*>(s_po + row * kPOStride + col + i);
                dst[0] = make_float4(o[0], o[1], o[2], o[3]);
                dst[1] = make_float4(o[4], o[5], o[6], o[7]);
                continue;
              }
              uint4 v;
              v.x = pack_bf16(o[0], o[1]);
              v.y = pack_bf16(o[2], o[3]);
              v.z = pack_bf16(o[4], o[5]);
              v.w = pack_bf16(o[6], o[7]);
              if (!kBoundsChecks || bounds_ok(dev_range(p.out, (size_t)p.Lq * p.H * kHD * 2), orow + col + i,
                                              sizeof(uint4), p.status))
                *reinterpret_cast<uint4*>(orow + col + i) = v;
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
  if (split) {
    // ---- split keys: combine the cluster's partials ----
    // Every CTA of the cluster passes both barriers, whatever happened above.
    cluster_sync();  // every CTA's partials are written and visible to the cluster
    // CTA `rank` writes rows [rank * rows, (rank + 1) * rows) of the tile:
    // out = sum_b 2^(m_b - M) O_b / sum_b 2^(m_b - M) l_b with M = max_b m_b.
    const int rows = kBM / csplit;
    for (int i = threadIdx.x; i < rows * (kHD / 8); i += kThreads) {
      const int row = rank * rows + i / (kHD / 8), c = (i % (kHD / 8)) * 8;
      const int q = q0 + row;
      if (q >= p.Lq) continue;
      float M = -INFINITY;
      for (int b = 0; b < csplit; ++b) M = fmaxf(M, ld_cluster(cluster_addr(s_pm + row, b)));
      float den = 0.f;
      float num[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (int b = 0; b < csplit; ++b) {
        const float w = ex2(ld_cluster(cluster_addr(s_pm + row, b)) - M);
        den = fmaf(w, ld_cluster(cluster_addr(s_pl + row, b)), den);
        const uint32_t src = cluster_addr(s_po + row * kPOStride + c, b);
        const float4 u0 = ld_cluster4(src), u1 = ld_cluster4(src + 16);
        num[0] = fmaf(w, u0.x, num[0]);
        num[1] = fmaf(w, u0.y, num[1]);
        num[2] = fmaf(w, u0.z, num[2]);
        num[3] = fmaf(w, u0.w, num[3]);
        num[4] = fmaf(w, u1.x, num[4]);
        num[5] = fmaf(w, u1.y, num[5]);
        num[6] = fmaf(w, u1.z, num[6]);
        num[7] = fmaf(w, u1.w, num[7]);
      }
      const float inv = 1.f / den;
      uint4 v;
      v.x = pack_bf16(num[0] * inv, num[1] * inv);
      v.y = pack_bf16(num[2] * inv, num[3] * inv);
      v.z = pack_bf16(num[4] * inv, num[5] * inv);
      v.w = pack_bf16(num[6] * inv, num[7] * inv);
      __nv_bfloat16* dst = p.out + ((size_t)q * p.H + h) * kHD + c;
      if (!kBoundsChecks || bounds_ok(dev_range(p.out, (size_t)p.Lq * p.H * kHD * 2), dst, sizeof(uint4), p.status))
        *reinterpret_cast<uint4*>(dst) = v;
    }
    cluster_sync();  // no CTA leaves while another still reads its shared memory
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

namespace {
// Diagnostic: one thread waits, through the kernels' own bounded wait, on an
// mbarrier that nothing arrives on; the wait gives up after `limit` cycles and
// the time-out is recorded in the status word, as in any kernel of the library.
__global__ void wait_selftest_kernel(unsigned int* status, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  if (!mbar_wait(b, 0, &abort_flag, limit)) atomicOr(status, kStatusTimeout);
}
}  // namespace

cudaError_t launch_wait_selftest(unsigned int* status, long long limit_cycles, cudaStream_t stream) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(status, limit_cycles);
  return cudaGetLastError();
}

cudaError_t launch_attend_bf16(const Geometry& g, const void* Kc, const void* Vc, int Lk, const void* Kcur,
                               const void* Vcur, int Lk2, const void* Q, void* out, int Lq, float scale,
                               unsigned int* status, cudaStream_t stream, char* err, size_t errlen) {
  if (g.D != kHD) {
    snprintf(err, errlen, "bf16 attention supports head_dim 128 only (got %d)", g.D);
    return cudaErrorNotSupported;
  }
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) {
    snprintf(err, errlen, "cuTensorMapEncodeTiled is unavailable from the driver");
    return cudaErrorNotSupported;
  }
  {
    // The shared-memory opt-in is a per-device setting: once per device, with it current.
    static PerDevice<char> smem_opt_in;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    char done = 0;
    if (!smem_opt_in.get(dev, [&e](int, char* v) {
          e = cudaFuncSetAttribute(attend_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
          if (e == cudaSuccess)
            e = cudaFuncSetAttribute(attend_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
          *v = 1;
          return e == cudaSuccess;
        }, &done))
      return e != cudaSuccess ? e : cudaErrorInvalidDevice;
  }
  AttnParams prm;
  const uint64_t row = (uint64_t)kHD * 2;
  // An absent source (Lk == 0 or Lk2 == 0) gets a valid one-row map that no tile reads.
  const void* k1 = Lk > 0 ? Kc : Q;
  const void* v1 = Lk > 0 ? Vc : Q;
  const void* k2 = Lk2 > 0 ? Kcur : Q;
  const void* v2 = Lk2 > 0 ? Vcur : Q;
  if (!encode_3d(enc, &prm.tmQ, Q, kHD, g.H, Lq, row, row * g.H, 64, 1, kBM) ||
      !encode_3d(enc, &prm.tmK, k1, kHD, Lk > 0 ? Lk : 1, g.H, row, row * g.M * g.N, 64, kBN, 1) ||
      !encode_3d(enc, &prm.tmV, v1, kHD, Lk > 0 ? Lk : 1, g.H, row, row * g.M * g.N, 64, kBN, 1) ||
      !encode_3d(enc, &prm.tmK2, k2, kHD, g.H, Lk2 > 0 ? Lk2 : 1, row, row * g.H, 64, 1, kBN) ||
      !encode_3d(enc, &prm.tmV2, v2, kHD, g.H, Lk2 > 0 ? Lk2 : 1, row, row * g.H, 64, 1, kBN)) {
    snprintf(err, errlen, "cuTensorMapEncodeTiled rejected a tensor map (Lq=%d Lk=%d Lk2=%d)", Lq, Lk, Lk2);
    return cudaErrorInvalidValue;
  }
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.Lq = Lq;
  prm.Lk = Lk;
  prm.Lk2 = Lk2;
  prm.H = g.H;
  prm.scale_log2 = scale * 1.4426950408889634f;
  prm.status = status;
  // One CTA per SM.  While the query tiles fill less than half the SMs (few
  // queries, or few heads), split each tile's keys over a cluster of 2, 4 or 8
  // CTAs (each keeping at least 4 key tiles), which combine their partials
  // through distributed shared memory.
  const long long tiles_q = (Lq + kBM - 1) / kBM;
  const long long ctas = tiles_q * g.H;
  const int n_all = (Lk + kBN - 1) / kBN + (Lk2 + kBN - 1) / kBN;
  const long long sms = current_device_sm_count(148);
  int csplit = 1;
  while (csplit < 8 && ctas * csplit * 2 <= sms && n_all >= 8 * csplit) csplit *= 2;
  // A cluster needs csplit SMs of one GPC with a CTA's shared memory free each:
  // take the largest size the device can place (looked up once per device).
  {
    static PerDevice<int> max_cluster;
    int dev = 0, fit = 1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    max_cluster.get(dev, [](int, int* v) {
      *v = 1;
      for (int c = 2; c <= 8; c *= 2) {
        cudaLaunchConfig_t oc = {};
        oc.gridDim = dim3((unsigned)c, 1);
        oc.blockDim = dim3(kThreads);
        oc.dynamicSmemBytes = kSmemBytes;
        cudaLaunchAttribute ca[1];
        ca[0].id = cudaLaunchAttributeClusterDimension;
        ca[0].val.clusterDim.x = (unsigned)c;
        ca[0].val.clusterDim.y = 1;
        ca[0].val.clusterDim.z = 1;
        oc.attrs = ca;
        oc.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, attend_tc_kernel<true>, &oc) != cudaSuccess || n < 1) {
          cudaGetLastError();  // clear a refused query; the smaller size stands
          break;
        }
        *v = c;
      }
      return true;
    }, &fit);
    while (csplit > fit) csplit /= 2;
  }
  prm.csplit = csplit;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(tiles_q * csplit), g.H);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)csplit;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = csplit > 1 ? 2 : 1;
  return csplit > 1 ? cudaLaunchKernelEx(&cfg, attend_tc_kernel<true>, prm)
                    : cudaLaunchKernelEx(&cfg, attend_tc_kernel<false>, prm);
}

}  // namespace fademem
