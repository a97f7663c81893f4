// Persistent bf16 GEMM on the 5th-generation tensor cores (tcgen05) of sm_103a:
//   out = A[M][K] @ W[N][K]^T   (both operands K-major, fp32 accumulation in TMEM)
// with the step's epilogues fused (RoPE on Q/K, residual add, SwiGLU, LM-head softmax
// partials).  These are the dense contractions of the denoise step's forward (the
// single bidirectional pass of Sec. 3.3 step (ii)).
//
// Structure (one CTA per SM, 192 threads):
//   warp 0 lane 0 : TMA producer.  Per 64-wide K block, one 128x64 A box and one
//                   BNx64 W box (128-byte swizzle) land in a STAGES-deep smem ring,
//                   completing a transaction-count mbarrier.
//   warp 1        : allocates TMEM (2 x BN fp32 columns: double-buffered accumulator);
//                   lane 0 issues tcgen05.mma (M=128, N=BN, K=16) x4 per K block and
//                   tcgen05.commit to release smem stages / publish finished tiles.
//   warps 2..5    : epilogue.  Warp w reads TMEM lanes 32*(w%4)..+31 (one output row
//                   per thread) with tcgen05.ld and applies the fused epilogue while the
//                   MMA warp accumulates the next tile into the other TMEM buffer.
// Tiles are visited M-fastest so the CTAs working on one weight tile run together and
// share it through L2.  Every mbarrier wait is bounded: on timeout the kernel records
// DERR_WAIT_TIMEOUT, lets the other roles leave, waits (bounded) for its own copies
// and MMAs in flight, frees TMEM and returns.
#include <cudaTypedefs.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace dcl {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // bf16 elements in one 128-byte swizzle row
constexpr int A_STAGE_BYTES = BM * BK * 2;
constexpr int NUM_THREADS = 192;

template <int BN>
struct Cfg {
  static constexpr int B_STAGE_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + 256;
};


__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* dst, const float* v) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    d4[i] = make_uint4(pack_bf16x2(v[8 * i + 0], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                       pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
}

// ------------------------------------------------------------------ epilogues
// (one-CTA tiles; the CTA-pair kernel has its own, staged through shared memory)
struct Parts {};  // no earlier partial sums: one-CTA tiles are never split

// Accumulator columns [col, col + 32) of this thread's row.
__device__ __forceinline__ void load_cols(uint32_t taddr, int col, float (&v)[32], const Parts&) {
  uint32_t r[32];
  tmem_ld32(taddr + col, r);
  tmem_ld_wait();
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = f32(r[i]);
}

// taddr: TMEM address of (this warp's first lane, accumulator column 0); row: output row
// of this thread; n_blk: tile column index.  All tcgen05.ld run warp-uniformly; only the
// stores are guarded by row < M.
template <int BN, int EPI>
__device__ __forceinline__ void epilogue_tile(uint32_t taddr, int row, int n_blk, int M, int N,
                                              const EpiParams& ep, const Parts& ps) {
  const int n0 = n_blk * BN;
  const bool live = row < M;
  if constexpr (EPI == EPI_BF16) {
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      load_cols(taddr, c, v, ps);
      if (live && n0 + c < N)
        store_bf16x32(reinterpret_cast<__nv_bfloat16*>(ep.out) + (size_t)row * ep.ldo + n0 + c, v);
    }
  } else if constexpr (EPI == EPI_RESID_F32) {
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      load_cols(taddr, c, v, ps);
      if (live && n0 + c < N) {
        float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(ep.out) +
                                                (size_t)row * ep.ldo + n0 + c);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float4 o = dst[i];
          o.x += v[4 * i + 0];
          o.y += v[4 * i + 1];
          o.z += v[4 * i + 2];
          o.w += v[4 * i + 3];
          dst[i] = o;
        }
      }
    }
  } else if constexpr (EPI == EPI_QKV_ROPE) {
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(ep.out) + (size_t)row * ep.ldo + n0;
    if (n0 < ep.rope_cols) {
      const int hd = ep.head_dim, half = hd >> 1;
      const int pos = live ? row % ep.seq_T : 0;
      const float* cs = ep.rope_cos + pos;  // [half][rope_T]: a warp's rows read one line
      const float* sn = ep.rope_sin + pos;
#pragma unroll 1
      for (int hb = 0; hb < BN; hb += hd) {
#pragma unroll 1
        for (int j0 = 0; j0 < half; j0 += 32) {
          float lo[32], hi[32];
          load_cols(taddr, hb + j0, lo, ps);
          load_cols(taddr, hb + half + j0, hi, ps);
          if (live) {
            float a[32], b[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const size_t jt = (size_t)(j0 + i) * ep.rope_T;
              const float c = __ldg(cs + jt), s = __ldg(sn + jt);
              a[i] = lo[i] * c - hi[i] * s;
              b[i] = hi[i] * c + lo[i] * s;
            }
            store_bf16x32(out + hb + j0, a);
            store_bf16x32(out + hb + half + j0, b);
          }
        }
      }
    } else {
#pragma unroll 1
      for (int c = 0; c < BN; c += 32) {
        float v[32];
        load_cols(taddr, c, v, ps);
        if (live) store_bf16x32(out + c, v);
      }
    }
  } else if constexpr (EPI == EPI_SWIGLU) {
    constexpr int H2 = BN / 2;
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(ep.out) + (size_t)row * ep.ldo + n_blk * H2;
#pragma unroll 1
    for (int c = 0; c < H2; c += 32) {
      float g[32], u[32];
      load_cols(taddr, c, g, ps);
      load_cols(taddr, H2 + c, u, ps);
      if (live) {
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = __fdividef(g[i], 1.0f + __expf(-g[i])) * u[i];
        store_bf16x32(out + c, v);
      }
    }
  } else if constexpr (EPI == EPI_LMHEAD) {
    // Online softmax over this tile's columns: running max m (= top-1 value), sum of
    // exp(z - m), argmax (lowest column on ties: columns arrive in increasing order and
    // only a strictly larger value replaces the leader), the second largest value, and
    // the entropy sum u = sum exp(z - m) * y with y = (z - m) log2(e).
    float m = -INFINITY, s = 0.f, t2 = -INFINITY, u = 0.f;
    int id = -1;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      load_cols(taddr, c, v, ps);
      const int col0 = n0 + c;
      float cm = m;
      int cid = id;
      float c2 = t2;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        if (col0 + i >= ep.vocab) v[i] = -INFINITY;
        if (v[i] > cm) {
          c2 = cm;
          cm = v[i];
          cid = col0 + i;
        } else if (v[i] > c2) {
          c2 = v[i];
        }
      }
      if (cm > -INFINITY) {
        const float mb = cm * kLog2e;
        const float d = m * kLog2e - mb;  // -inf before the first live column
        const float al = exp2f(d);
        float acc = s * al;
        float accu = s > 0.f ? al * fmaf(d, s, u) : 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float y = fmaf(v[i], kLog2e, -mb);
          const float e = exp2f(y);
          acc += e;
          accu = fmaf(e, fmaxf(y, -200.f), accu);  // e = 0 below -149: the term's limit 0
        }
        s = acc;
        u = accu;
      }
      m = cm;
      id = cid;
      t2 = c2;
    }
    if (live) {
      const int nblk = (N + BN - 1) / BN;
      float4* part = reinterpret_cast<float4*>(ep.out);
      part[(size_t)row * nblk + n_blk] = make_float4(m, s, __int_as_float(id), t2);
      if (ep.ent_part) ep.ent_part[(size_t)row * nblk + n_blk] = u;
    }
  }
}

// ------------------------------------------------------------------ the kernel
template <int BN, int EPI>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmb,
                   int M, int N, int K, EpiParams ep, int* err) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  const uint32_t sA = base;
  const uint32_t sB = base + C::STAGES * A_STAGE_BYTES;
  const uint32_t bars = sB + C::STAGES * C::B_STAGE_BYTES;
  const uint32_t full0 = bars;                       // full[s]   = full0 + 8 s
  const uint32_t empty0 = bars + 8 * C::STAGES;      // empty[s]  = empty0 + 8 s
  const uint32_t tfull0 = bars + 16 * C::STAGES;     // tfull[ab] = tfull0 + 8 ab
  const uint32_t tempty0 = tfull0 + 16;              // tempty[ab]
  const uint32_t drain = tempty0 + 16;
  const uint32_t holder = drain + 8;
  volatile uint32_t* holder_ptr = reinterpret_cast<volatile uint32_t*>(smem + (holder - base));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + (holder + 4 - base));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_m = (M + BM - 1) / BM;
  const int num_n = (N + BN - 1) / BN;
  const int num_tiles = num_m * num_n;
  const int num_kb = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(tfull0, 1);
    mbar_init(tfull0 + 8, 1);
    mbar_init(tempty0, 128);
    mbar_init(tempty0 + 8, 128);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tma);
    prefetch_tmap(&tmb);
  }
  if (warp == 1) tmem_alloc(holder, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *holder_ptr;
  pdl_wait();  // the previous kernel of the step has completed
  pdl_launch_dependents();

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      long issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x) {
        const int m_blk = t % num_m, n_blk = t / num_m;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full0 + 8 * stage, C::STAGE_BYTES);
          tma_load_2d(sA + stage * A_STAGE_BYTES, &tma, kb * BK, m_blk * BM, full0 + 8 * stage);
          tma_load_2d(sB + stage * C::B_STAGE_BYTES, &tmb, kb * BK, n_blk * BN, full0 + 8 * stage);
          ++issued;
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
        // wait (bounded) until every copy this thread issued has landed
        for (int s = 0; s < C::STAGES && s < issued; ++s) {
          const long arms = (issued - 1 - s) / C::STAGES + 1;
          volatile int no_abort = 0;
          mbar_wait(full0 + 8 * s, (uint32_t)((arms - 1) & 1), &no_abort);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t idesc = make_idesc(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int j = 0;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x, ++j) {
        const int ab = j & 1;
        const uint32_t aph = (uint32_t)(j >> 1) & 1u;
        if (!mbar_wait(tempty0 + 8 * ab, aph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          const uint64_t da = sw128_desc(sA + stage * A_STAGE_BYTES);
          const uint64_t db = sw128_desc(sB + stage * C::B_STAGE_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)  // advance 16 elements = 32 bytes = 2 desc units
            umma_bf16(d_tmem, da + 2 * k, db + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          umma_commit(empty0 + 8 * stage);
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(tfull0 + 8 * ab);
      }
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
      }
      // all MMAs issued by this thread complete before TMEM is released
      umma_commit(drain);
      volatile int no_abort = 0;
      mbar_wait(drain, 0, &no_abort);
    }
  } else {
    // ------------------------------------------------ epilogue warps 2..5
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    int j = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++j) {
      const int ab = j & 1;
      const uint32_t aph = (uint32_t)(j >> 1) & 1u;
      if (!mbar_wait(tfull0 + 8 * ab, aph, abort_flag)) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
        break;
      }
      tc_fence_after();
      const int m_blk = t % num_m, n_blk = t / num_m;
      const int row = m_blk * BM + q * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN);
      epilogue_tile<BN, EPI>(taddr, row, n_blk, M, N, ep, Parts{});
      tc_fence_before();
      mbar_arrive(tempty0 + 8 * ab);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ 2-CTA variant
// A CTA pair (cluster of 2) computes a 256 x 256 tile with tcgen05.mma.cta_group::2:
// each CTA stages its own 128 rows of A and its own 128-row half of the weight tile
// (32 KB per 64-wide K block instead of 48 KB), the even CTA issues the M = 256 MMAs for
// both, and each CTA's TMEM receives its 128 rows x 256 columns.  A ring stage holds KA2
// K blocks (KA2 x 4 MMAs per stage barrier round trip).
//
// The epilogue leaves through TMA: each epilogue warp owns 32 output rows and two 4 KB
// staging boxes (32 rows x 128 bytes, 128-byte swizzle, so that one row per thread is
// written without bank conflicts); a box is stored (bf16 / fp32 outputs) or added into
// the fp32 residual stream (cp.reduce.async.bulk .add) by one lane while the warp fills
// the other box.  Whole 128-byte row segments reach L2 instead of 16-byte pieces of 32
// different rows.
#ifndef DCL_PAIR_KA
#define DCL_PAIR_KA 1
#endif
constexpr int KA2 = DCL_PAIR_KA;
constexpr int A2_STAGE_BYTES = KA2 * A_STAGE_BYTES;
constexpr int B2_BLOCK_BYTES = 128 * BK * 2;
constexpr int B2_STAGE_BYTES = KA2 * B2_BLOCK_BYTES;
constexpr int STAGE2_BYTES = A2_STAGE_BYTES + B2_STAGE_BYTES;
constexpr int STAGES2 = (6 * 32768) / STAGE2_BYTES;
constexpr int RING2_BYTES = STAGES2 * STAGE2_BYTES;
constexpr int BOX_BYTES = 32 * 128;                 // one staging box: 32 rows x 128 bytes
constexpr int STG2_BYTES = 4 * 2 * BOX_BYTES;       // 4 epilogue warps x 2 boxes
constexpr int FIX_BOXES = RING2_BYTES / (4 * BOX_BYTES);  // stream-K fix-up boxes per warp
constexpr int BARS2_BYTES = 768;
static_assert(16 * STAGES2 + 48 + 8 * 4 * FIX_BOXES + 8 + 8 * 16 <= BARS2_BYTES, "barrier area");
static_assert(FIX_BOXES >= 2, "fix-up needs two boxes per warp");
constexpr size_t SMEM2 = 1024 + (size_t)RING2_BYTES + STG2_BYTES + BARS2_BYTES;
static_assert(SMEM2 <= 232448, "shared memory per CTA");
constexpr int TMEM2_COLS = 512;
// DSMEM split: the received fp32 half sum moves in 64-column chunks per 32-row band, each
// a contiguous block of 32 rows padded by 16 bytes (eight lanes' 16-byte accesses to
// eight consecutive rows fall in distinct bank groups), block (band, chunk) at
// (band * 4 + chunk) * DS_BLOCK_BYTES
constexpr int DS_ROW_BYTES = 64 * 4 + 16;
constexpr int DS_BLOCK_BYTES = 32 * DS_ROW_BYTES;
static_assert(16 * DS_BLOCK_BYTES <= RING2_BYTES, "the received sum lives in the operand ring");

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm, int x, int y,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(holder), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive (once) on the mbarrier at this offset in every CTA of cta_mask
__device__ __forceinline__ void umma_commit_pair(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          bar),
      "h"(cta_mask)
      : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// Bulk copy of `bytes` (a multiple of 16) from this CTA's shared memory to another CTA's
// (dst and bar: shared::cluster addresses from mapa), completing on that CTA's barrier.
__device__ __forceinline__ void bulk_copy_to_cluster(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "r"(src), "r"(bytes), "r"(bar)
      : "memory");
}
// Bounded wait for a phase completed by arrivals released at cluster scope (data that
// other CTAs of the cluster wrote into this CTA's shared memory is visible afterwards).
__device__ __forceinline__ bool mbar_try_wait_acq_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}
__device__ __noinline__ bool mbar_wait_acq_cluster(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait_acq_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (;;) {
    if (mbar_try_wait_acq_cluster(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
// This lane's row of a staging box: 32 fp32 values, or 32 bf16 values into half h
// (columns 32h .. 32h + 31) of a 64-column bf16 box.
__device__ __forceinline__ void stage_f32(uint32_t box, int lane, const float (&v)[32]) {
#pragma unroll
  for (int k = 0; k < 8; ++k)
    st_shared_v4(box + swz(lane, k), __float_as_uint(v[4 * k]), __float_as_uint(v[4 * k + 1]),
                 __float_as_uint(v[4 * k + 2]), __float_as_uint(v[4 * k + 3]));
}
__device__ __forceinline__ void stage_bf16(uint32_t box, int lane, int h, const float (&v)[32]) {
#pragma unroll
  for (int k = 0; k < 4; ++k)
    st_shared_v4(box + swz(lane, 4 * h + k), pack_bf16x2(v[8 * k], v[8 * k + 1]), pack_bf16x2(v[8 * k + 2], v[8 * k + 3]),
                 pack_bf16x2(v[8 * k + 4], v[8 * k + 5]), pack_bf16x2(v[8 * k + 6], v[8 * k + 7]));
}

// One epilogue warp's output stream: its 32-row band and its two staging boxes.
struct Stage {
  uint32_t box0;   // shared address of this warp's first box (the second follows)
  int lane;
  int row0;        // first output row of the band
  bool live;       // row0 < M (a band wholly below M is not stored)
  int n;           // boxes issued so far (selects the box)
  // a free box: the one issued two boxes ago has been read
  __device__ __forceinline__ uint32_t acquire() {
    if (lane == 0) bulk_wait_read<1>();
    __syncwarp();
    return box0 + (uint32_t)(n & 1) * BOX_BYTES;
  }
  // issue the box just filled: a store (or reduce-add) of it at column x of the band
  __device__ __forceinline__ void issue(const CUtensorMap* tm, uint32_t box, int x, int y, bool reduce) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (live) {
        if (reduce)
          tma_reduce_add_2d(tm, box, x, y);
        else
          tma_store_2d(tm, box, x, y);
      }
      bulk_commit();
    }
    ++n;
  }
  // the same for a box of a 3-D tensor (x, y, z)
  __device__ __forceinline__ void issue3(const CUtensorMap* tm, uint32_t box, int x, int y, int z) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (live) tma_store_3d(tm, box, x, y, z);
      bulk_commit();
    }
    ++n;
  }
  // every store issued so far has completed and is ordered before later generic
  // accesses of this warp (before a release that publishes it)
  __device__ __forceinline__ void drain() {
    if (lane == 0) {
      bulk_wait_all();
      fence_proxy_async_global();
    }
    __syncwarp();
  }
};

// Accumulator (plus earlier partials) of this warp's 32 rows x 32 columns at col.
struct Src {
  uint32_t taddr;        // this warp's TMEM lanes, accumulator column 0
  bool has_sum = false;  // TMEM at tsum holds the summed earlier stream-K partials
  uint32_t tsum = 0;     // (TMEM address 0 is a valid address)
  const float* part = nullptr;  // split-K: earlier splits' partials, row-major [rows][256]
  size_t part_stride = 0;       // floats between consecutive splits' partials
  int nparts = 0;
  int row = 0;                  // this thread's row within the CTA's 128-row half
  uint32_t dpart = 0;           // DSMEM split: the other K half's sum in this CTA's shared
                                // memory, in (band, chunk) blocks (0: none)
  uint32_t dbar = 0;            // DSMEM split: this band's 4 chunk barriers
  mutable uint32_t dready = 0;  // chunks waited for so far
  volatile int* dabort = nullptr;
  int* derr = nullptr;
};
// DSMEM split: the received 64-column chunk has arrived (bounded wait, once per chunk;
// warp-uniform)
__device__ __forceinline__ void ds_chunk_ready(const Src& s, int chunk) {
  if (s.dready & (1u << chunk)) return;
  if (!mbar_wait_acq_cluster(s.dbar + 8 * chunk, 0, s.dabort)) {
    *s.dabort = 1;
    report_error(s.derr, DERR_WAIT_TIMEOUT);
  }
  s.dready |= 1u << chunk;
}
__device__ __forceinline__ void src_cols(const Src& s, int col, float (&v)[32]) {
  uint32_t r[32];
  tmem_ld32(s.taddr + col, r);
  if (s.dpart) {
    ds_chunk_ready(s, col >> 6);
    tmem_ld_wait();
    const uint32_t a = s.dpart + (uint32_t)((((s.row >> 5) * 4 + (col >> 6)) * 32 + (s.row & 31)) * DS_ROW_BYTES +
                                            (col & 63) * 4);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 t = ld_shared_v4(a + 16 * k);
      v[4 * k] = f32(r[4 * k]) + t.x;  // K lower half (own) + K upper half (received)
      v[4 * k + 1] = f32(r[4 * k + 1]) + t.y;
      v[4 * k + 2] = f32(r[4 * k + 2]) + t.z;
      v[4 * k + 3] = f32(r[4 * k + 3]) + t.w;
    }
  } else if (s.has_sum) {
    uint32_t q[32];
    tmem_ld32(s.tsum + col, q);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = f32(q[i]) + f32(r[i]);
  } else if (s.nparts > 0) {
    tmem_ld_wait();
    const float4* q = reinterpret_cast<const float4*>(s.part + (size_t)s.row * 256 + col);
    float a[32];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 t = __ldcg(q + k);
      a[4 * k] = t.x, a[4 * k + 1] = t.y, a[4 * k + 2] = t.z, a[4 * k + 3] = t.w;
    }
    for (int sp = 1; sp < s.nparts; ++sp) {
      const float4* qs = reinterpret_cast<const float4*>(s.part + sp * s.part_stride + (size_t)s.row * 256 + col);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float4 t = __ldcg(qs + k);
        a[4 * k] += t.x, a[4 * k + 1] += t.y, a[4 * k + 2] += t.z, a[4 * k + 3] += t.w;
      }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = a[i] + f32(r[i]);
  } else {
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = f32(r[i]);
  }
}

// Accumulator columns [c, c + 64) of the band as one bf16 box at output column x.
__device__ __forceinline__ void store_bf16_box(const Src& s, Stage& o, const CUtensorMap* tmc, int c, int x) {
  const uint32_t b = o.acquire();
#pragma unroll 1
  for (int h = 0; h < 2; ++h) {
    float v[32];
    src_cols(s, c + 32 * h, v);
    stage_bf16(b, o.lane, h, v);
  }
  o.issue(tmc, b, x, o.row0, false);
}

// The fused epilogues of a pair tile (256 rows x W columns: W = 256, or 128 for piece
// `piece` of a tile cut in two), for one warp's 32-row band of one CTA half.  A piece
// covers output columns [n_blk * 256 + piece * W, + W); with SwiGLU it holds W/2 gate
// columns and the W/2 matching up columns.  All tcgen05.ld run warp-uniformly.
template <int EPI>
__device__ __forceinline__ void epilogue_pair(const Src& s, Stage& o, const CUtensorMap* tmc, const CUtensorMap* tmv,
                                              const CUtensorMap* tmk, int row, int n_blk, int M, int N,
                                              const EpiParams& ep, int piece = 0, int W = 256) {
  const int n0 = n_blk * 256 + piece * W;
  if constexpr (EPI == EPI_BF16) {
#pragma unroll 1
    for (int c = 0; c < W && n0 + c < N; c += 64) store_bf16_box(s, o, tmc, c, n0 + c);
  } else if constexpr (EPI == EPI_RESID_F32) {
#pragma unroll 1
    for (int c = 0; c < W; c += 32) {
      float v[32];
      src_cols(s, c, v);
      if (n0 + c >= N) break;
      const uint32_t b = o.acquire();
      stage_f32(b, o.lane, v);
      o.issue(tmc, b, n0 + c, o.row0, true);
    }
  } else if constexpr (EPI == EPI_QKV_ROPE) {
    // the band's sequence and first position (32 consecutive positions of one sequence)
    int bz = 0, t0 = 0;
    if (o.live) {
      bz = ep.row_seq ? ep.row_seq[o.row0] : o.row0 / ep.seq_T;
      t0 = ep.row_pos ? ep.row_pos[o.row0] : o.row0 - bz * ep.seq_T;
    }
    if (n0 < ep.rope_cols) {
      const int hd = ep.head_dim, half = hd >> 1;
      const int pos = row < M ? (ep.row_pos ? ep.row_pos[row] : row % ep.seq_T) : 0;
      const bool to_k = ep.k_store && n0 >= ep.k_col0;  // k columns go to the key store
      // tables [half][rope_T]: the 32 consecutive positions of a band read one 128-byte line
      const float* cs = ep.rope_cos + pos;
      const float* sn = ep.rope_sin + pos;
#pragma unroll 1
      for (int hb = 0; hb < W; hb += hd) {
        // rotate-half pairs (j, j + half).  hd 128: box `part` 0 holds the rotated columns
        // [hb, hb + 64) = x_j c - x_{j+64} s, part 1 holds [hb + 64, hb + 128) = x_{j+64} c
        // + x_j s; each part re-reads both source halves from TMEM so that one box at a
        // time is staged and the stores stay pipelined (a head never waits for every store
        // in flight, which under a concurrent mainloop cost ~20 us per tile).  hd 64: one
        // box [hb, hb + 64) holds both halves.
        const int nparts = hd == 128 ? 2 : 1;
#pragma unroll 1
        for (int part = 0; part < nparts; ++part) {
          const uint32_t b = o.acquire();
#pragma unroll 1
          for (int j0 = 0; j0 < half; j0 += 32) {
            float lo[32], hi[32];
            src_cols(s, hb + j0, lo);
            src_cols(s, hb + half + j0, hi);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const size_t jt = (size_t)(j0 + i) * ep.rope_T;
              const float c = __ldg(cs + jt), sv = __ldg(sn + jt);
              const float x = lo[i], y = hi[i];
              lo[i] = x * c - y * sv;
              hi[i] = y * c + x * sv;
            }
            if (hd == 128) {
              stage_bf16(b, o.lane, j0 >> 5, part == 0 ? lo : hi);
            } else {
              stage_bf16(b, o.lane, 0, lo);
              stage_bf16(b, o.lane, 1, hi);
            }
          }
          if (to_k)
            o.issue3(tmk, b, n0 + hb + 64 * part - ep.k_col0, t0, bz);
          else
            o.issue(tmc, b, n0 + hb + 64 * part, o.row0, false);
        }
      }
    } else if (ep.vt_heads > 0) {
      // v columns leave transposed, as the attention's K-major operand: boxes of 64
      // channels x 32 tokens of vt [batch * G][hd][T], in fp16 (the attention multiplies P in
      // fp16 by them; the bf16-rounded v is held exactly)
#pragma unroll 1
      for (int c = 0; c < W && n0 + c < N; c += 64) {
        const int cv = n0 + c - ep.rope_cols, g = cv / ep.head_dim, d0 = cv - g * ep.head_dim;
        const uint32_t b = o.acquire();
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          float v[32];
          src_cols(s, c + 32 * h, v);
#pragma unroll
          for (int e = 0; e < 32; ++e)
            st_shared_u16(b + (uint32_t)((32 * h + e) * 64 + 2 * o.lane),
                          __half_as_ushort(__float2half_rn(__bfloat162float(__float2bfloat16_rn(v[e])))));
        }
        o.issue3(tmv, b, t0, d0, bz * ep.vt_heads + g);
      }
    } else {
#pragma unroll 1
      for (int c = 0; c < W && n0 + c < N; c += 64) store_bf16_box(s, o, tmc, c, n0 + c);
    }
  } else if constexpr (EPI == EPI_SWIGLU) {
    // columns [0, W/2) of the tile are gate rows, [W/2, W) the matching up rows
    const int G2 = W >> 1;
#pragma unroll 1
    for (int c = 0; c < G2; c += 64) {
      const uint32_t b = o.acquire();
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        float g[32], u[32];
        src_cols(s, c + 32 * h, g);
        src_cols(s, G2 + c + 32 * h, u);
        float v[32];
#pragma unroll
        // silu(g) * u with the SFU's exp2 and reciprocal (a few fp32 ulp, far below the
        // output's bf16 rounding); the IEEE division here cost ~6 us per tile
        for (int i = 0; i < 32; ++i) v[i] = __fdividef(g[i], 1.0f + __expf(-g[i])) * u[i];
        stage_bf16(b, o.lane, h, v);
      }
      o.issue(tmc, b, n_blk * 128 + piece * G2 + c, o.row0, false);
    }
  } else if constexpr (EPI == EPI_LMHEAD) {
    // Online softmax over this tile's columns (see epilogue_tile); one float4 per row.
    float m = -INFINITY, sum = 0.f, t2 = -INFINITY, u = 0.f;
    int id = -1;
#pragma unroll 1
    for (int c = 0; c < 256; c += 32) {
      float v[32];
      src_cols(s, c, v);
      const int col0 = n0 + c;
      float cm = m;
      int cid = id;
      float c2 = t2;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        if (col0 + i >= ep.vocab) v[i] = -INFINITY;
        if (v[i] > cm) {
          c2 = cm;
          cm = v[i];
          cid = col0 + i;
        } else if (v[i] > c2) {
          c2 = v[i];
        }
      }
      if (cm > -INFINITY) {
        const float mb = cm * kLog2e;
        const float d = m * kLog2e - mb;  // -inf before the first live column
        const float al = exp2f(d);
        float acc = sum * al;
        float accu = sum > 0.f ? al * fmaf(d, sum, u) : 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float y = fmaf(v[i], kLog2e, -mb);
          const float e = exp2f(y);
          acc += e;
          accu = fmaf(e, fmaxf(y, -200.f), accu);  // e = 0 below -149: the term's limit 0
        }
        sum = acc;
        u = accu;
      }
      m = cm;
      id = cid;
      t2 = c2;
    }
    if (row < M) {
      const int nblk = (N + 255) / 256;
      float4* part = reinterpret_cast<float4*>(ep.out);
      part[(size_t)row * nblk + n_blk] = make_float4(m, sum, __int_as_float(id), t2);
      if (ep.ent_part) ep.ent_part[(size_t)row * nblk + n_blk] = u;
    }
  }
}

// This warp's 32 rows x 256 columns of the accumulator, stored as an fp32 partial
// (rows y0 .. y0 + 31 of the workspace, [rows][256]).
__device__ __forceinline__ void store_partial_pair(const Src& s, Stage& o, const CUtensorMap* tmw, int y0) {
  const bool live = o.live;
  o.live = true;  // partials are stored for every band
#pragma unroll 1
  for (int c = 0; c < 256; c += 32) {
    float v[32];
    src_cols(s, c, v);
    const uint32_t b = o.acquire();
    stage_f32(b, o.lane, v);
    o.issue(tmw, b, c, y0, false);
  }
  o.live = live;
}

__device__ __forceinline__ void epilogue_bar() {  // the 128 epilogue threads (warps 2..5)
  asm volatile("bar.sync 1, 128;" ::: "memory");
}
// Bounded wait until the counter at f reaches target; false on timeout or abort.
__device__ __noinline__ bool wait_flag_geq(const int* f, int target, volatile int* abort_flag) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(f) : "memory");
  if (v >= target) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(100);
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(f) : "memory");
    if (v >= target) return true;
    if ((it & 15u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer() - t0 > kWaitLimitNs) return false;
    }
  }
}

// Stream-K fix-up, per epilogue warp.  A tile's last K segment is its CTA pair's last
// work item, so when it is reached the operand ring is idle in both CTAs and the second
// TMEM accumulator is free.  Each warp streams the n earlier partials of its 32 rows
// through FIX_BOXES boxes of its quarter of the ring (TMA loads of 32 rows x 32 fp32,
// 128-byte swizzle; column-chunk-major, partial-minor), sums each element in K order
// p0 + p1 + ... and writes the sum to TMEM at tsum, for the epilogue to add its own
// accumulator last.  Returns false (with *abort_flag set) if a box did not arrive in time;
// the result is warp-uniform.
__device__ __noinline__ bool fixup_to_tmem(const CUtensorMap* tmw, int y0, int slot_rows, int n, uint32_t ring,
                                           uint32_t bar0, uint32_t tsum, int lane, volatile int* abort_flag,
                                           int* err) {
  const int total = 8 * n;
  if (lane == 0) {
    fence_proxy_async_global();  // the partials were published to this CTA (acquire + barrier)
    for (int p = 0; p < total && p < FIX_BOXES; ++p) {
      mbar_arrive_expect_tx(bar0 + 8 * p, BOX_BYTES);
      tma_load_2d(ring + p * BOX_BYTES, tmw, (p / n) * 32, y0 + (p % n) * slot_rows, bar0 + 8 * p);
    }
  }
  bool ok = true;
#pragma unroll 1
  for (int j = 0; j < 8; ++j) {
    float a[32];
#pragma unroll 1
    for (int sl = 0; sl < n; ++sl) {
      const int p = j * n + sl, b = p % FIX_BOXES;
      if (ok && !mbar_wait(bar0 + 8 * b, (uint32_t)(p / FIX_BOXES) & 1u, abort_flag)) ok = false;
      ok = __all_sync(0xffffffffu, ok);
      if (ok) {
        const uint32_t box = ring + b * BOX_BYTES;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float4 t = ld_shared_v4(box + swz(lane, k));
          if (sl == 0) {
            a[4 * k] = t.x, a[4 * k + 1] = t.y, a[4 * k + 2] = t.z, a[4 * k + 3] = t.w;
          } else {
            a[4 * k] += t.x, a[4 * k + 1] += t.y, a[4 * k + 2] += t.z, a[4 * k + 3] += t.w;
          }
        }
      }
      fence_proxy_async_smem();  // this lane's reads of box b before its refill
      __syncwarp();
      const int nxt = p + FIX_BOXES;
      if (lane == 0 && ok && nxt < total) {
        mbar_arrive_expect_tx(bar0 + 8 * b, BOX_BYTES);
        tma_load_2d(ring + b * BOX_BYTES, tmw, (nxt / n) * 32, y0 + (nxt % n) * slot_rows, bar0 + 8 * b);
      }
    }
    if (ok) tmem_st32(tsum + j * 32, a);
  }
  tmem_st_wait();
  if (!ok) {
    *abort_flag = 1;
    report_error(err, DERR_WAIT_TIMEOUT);
  }
  return ok;
}

// ---- work items of a CTA pair ------------------------------------------------------
// A work item is a tile and a range [ku0, ku1) of its K units (KA2 K blocks each).
//   plain    : pair c takes tiles c, c + C, ...  (C pairs)
//   split-K  : items w = split * tiles + tile (split-major), pair c takes w = c, c + C, ...
//   stream-K : the first (tiles / C) * C tiles as plain rounds; the R left-over tiles'
//              R * U K units are then cut into Csk <= C equal contiguous ranges, one for
//              each of the first Csk pairs (Csk = 2R: every left-over tile in two halves).
//              A range covers the tail of one tile and/or the head of the next; the pair
//              processes the head first (it only writes a partial) and the tail second
//              (the tile's last segment: it waits for the other segments' partials, sums
//              them in K order and runs the epilogue), so no pair waits on a pair that is
//              itself waiting.
enum ItemKind : int { IT_PLAIN = 0, IT_SPLIT = 1, IT_PART = 2, IT_LAST = 3, IT_DS_RECV = 4, IT_DS_SEND = 5 };
struct Sched {
  int tiles, ku, C, splits;
  int fuse;     // 1: after the tiles, the second GEMM's tiles2 x splits2 K-split items (fused MLP)
  int tiles2, ku2, splits2;
  int streamk;  // 0: off; else the number of pairs (<= C) that share the left-over tiles
  int halves;   // 1: the tiles of a partial last round run as two 256 x 128 pieces each
  int ds;       // 1: the tiles of a partial last round are split by K over the two pairs
                //    of a 4-CTA cluster, the upper half's sum sent through DSMEM
};
struct Item {
  int t, ku0, ku1, kind;
  int g = 0;                   // fused MLP: 0 the first GEMM (gate/up), 1 the second (down)
  int piece = 0, width = 256;  // columns [piece * width, + width) of tile t
  int sp;     // IT_SPLIT: split index
  int rel;    // IT_PART / IT_LAST: stream-K tile index (0..R-1)
  int slot;   // IT_PART: partial slot; IT_LAST: number of earlier segments
};

__device__ __forceinline__ bool next_item(int idx, const Sched& s, int c, Item& it) {
  it.piece = 0;
  it.width = 256;
  it.g = 0;
  if (s.fuse) {
    // round robin over one sequence: the first GEMM's tiles (M-fastest), then the second's
    // K-split items, split-major (split s of every tile, M-fastest, before split s + 1):
    // split s reads the act columns that the first GEMM's tiles of column range s wrote,
    // which come early in the first sequence, so the items rarely wait
    const long w = (long)c + (long)idx * s.C;
    if (w < s.tiles) {
      it.t = (int)w;
      it.ku0 = 0;
      it.ku1 = s.ku;
      it.kind = IT_PLAIN;
      return true;
    }
    const long w2 = w - s.tiles;
    if (w2 >= (long)s.tiles2 * s.splits2) return false;
    it.g = 1;
    it.sp = (int)(w2 / s.tiles2);
    it.t = (int)(w2 % s.tiles2);
    it.ku0 = (int)((long)it.sp * s.ku2 / s.splits2);
    it.ku1 = (int)((long)(it.sp + 1) * s.ku2 / s.splits2);
    it.kind = IT_SPLIT;
    return true;
  }
  if (s.ds) {
    // c = pair index (pairs 2k and 2k + 1 form cluster k): full rounds of whole tiles,
    // then left-over tile `first + k` on cluster k, K lower half on its first pair (which
    // receives the other half's sum and runs the epilogue), upper half on its second
    const int full = s.tiles / s.C;
    if (idx < full) {
      it.t = c + idx * s.C;
      it.ku0 = 0;
      it.ku1 = s.ku;
      it.kind = IT_PLAIN;
      return true;
    }
    const int first = full * s.C, k = c >> 1;
    if (2 * (s.tiles - first) > s.C) {  // (fewer rows than planned) more left-over tiles
      it.t = c + idx * s.C;            // than clusters: whole tiles, round robin
      it.ku0 = 0;
      it.ku1 = s.ku;
      it.kind = IT_PLAIN;
      return it.t < s.tiles;
    }
    if (idx > full || first + k >= s.tiles) return false;
    it.t = first + k;
    const int mid = s.ku >> 1;
    const bool upper = (c & 1) != 0;
    it.ku0 = upper ? mid : 0;
    it.ku1 = upper ? s.ku : mid;
    it.kind = upper ? IT_DS_SEND : IT_DS_RECV;
    return true;
  }
  if (s.halves) {
    // full rounds of whole tiles, then every left-over tile as two half-width pieces on
    // two consecutive pairs (same rows of A, neighbouring rows of W): the last round
    // takes half as long and the pieces need no combination
    const int full = s.tiles / s.C;
    it.ku0 = 0;
    it.ku1 = s.ku;
    it.kind = IT_PLAIN;
    if (idx < full) {
      it.t = c + idx * s.C;
      return true;
    }
    const int first = full * s.C;
    const long w = (long)c + (long)(idx - full) * s.C;
    if (w >= 2L * (s.tiles - first)) return false;
    it.t = first + (int)(w >> 1);
    it.piece = (int)(w & 1);
    it.width = 128;
    return true;
  }
  if (s.splits > 1) {
    const long w = (long)c + (long)idx * s.C;
    if (w >= (long)s.tiles * s.splits) return false;
    it.sp = (int)(w / s.tiles);
    it.t = (int)(w % s.tiles);
    it.ku0 = (int)((long)it.sp * s.ku / s.splits);
    it.ku1 = (int)((long)(it.sp + 1) * s.ku / s.splits);
    it.kind = IT_SPLIT;
    return true;
  }
  const int rounds = s.streamk ? s.tiles / s.C : (s.tiles + s.C - 1) / s.C;
  if (idx < rounds) {
    it.t = c + idx * s.C;
    if (it.t >= s.tiles) return false;
    it.ku0 = 0;
    it.ku1 = s.ku;
    it.kind = IT_PLAIN;
    return true;
  }
  if (!s.streamk || c >= s.streamk) return false;
  const int first = rounds * s.C;
  const long RU = (long)(s.tiles - first) * s.ku;
  const long lo = (long)c * RU / s.streamk, hi = (long)(c + 1) * RU / s.streamk;
  if (hi <= lo) return false;
  const int ta = (int)(lo / s.ku), tb = (int)((hi - 1) / s.ku);
  const int k = idx - rounds;
  int rel, k0, k1;
  if (ta == tb) {
    if (k > 0) return false;
    rel = ta;
    k0 = (int)(lo - (long)ta * s.ku);
    k1 = (int)(hi - (long)ta * s.ku);
  } else if (k == 0) {  // head of the later tile first
    rel = tb;
    k0 = 0;
    k1 = (int)(hi - (long)tb * s.ku);
  } else if (k == 1) {  // then the tail of the earlier tile
    rel = ta;
    k0 = (int)(lo - (long)ta * s.ku);
    k1 = s.ku;
  } else {
    return false;
  }
  const int c_first = (int)((((long)rel * s.ku + 1) * s.streamk - 1) / RU);  // owner of the tile's first unit
  it.t = first + rel;
  it.rel = rel;
  it.ku0 = k0;
  it.ku1 = k1;
  it.kind = (k1 == s.ku) ? IT_LAST : IT_PART;
  it.slot = c - c_first;
  return true;
}

// Work items are taken in the order above by the producer, the MMA issuer and the
// epilogue alike.  Combination rules, all bit-reproducible:
//   split-K, residual epilogue: split s adds its accumulator to h after split s-1 has
//     (a per-tile counter, released by each split and reset by the last);
//   split-K, other epilogues: splits < S-1 store fp32 partials, the last split waits for
//     all of them, sums them in order with its own accumulator and runs the epilogue;
//   stream-K: as split-K's second rule, per left-over tile, the sum formed in TMEM.
// Partials are fp32 [rows][256] in the workspace: row ((tile * S + slot) * 2 + rank) * 128
// + r holds row r of CTA `rank`'s half of the tile (S slots per tile).  Items that are
// waited on never wait themselves before they publish, and every CTA is resident (grid <=
// SMs, one CTA per SM), so every wait ends.
//
// FUSE (the fused MLP, gemm_plan_mlp): the item sequence continues past the first GEMM's
// tiles with the second GEMM's K-split items (A = ta2, W = tb2, out = tc2 / ep2, N2 x K2,
// splits2 splits added to the residual in split order).  flags then holds, from the plan's
// row-block count num_m_max = ceil(M / 256): [num_m_max * num_n2 * 2] ordered-add counters,
// [num_m_max * splits2] readiness counters (each first-GEMM tile, when its act stores have
// completed, adds 1 per CTA to every split its 128 act columns fall in) and [num_m_max *
// splits2] pass counters (the last CTA to pass a readiness wait zeroes both for the next
// launch).  Every CTA is resident and a second-GEMM item waits only on first-GEMM tiles
// earlier in the sequence, which resident pairs have taken, so every wait ends.
template <int EPI, bool DS, bool FUSE = false>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmb,
                    const __grid_constant__ CUtensorMap tmbh, const __grid_constant__ CUtensorMap tmc,
                    const __grid_constant__ CUtensorMap tmw, const __grid_constant__ CUtensorMap tmv,
                    const __grid_constant__ CUtensorMap tmk, int M, int N, int K, EpiParams ep, int splits,
                    int streamk, int halves, int ws_slots, int* flags, float* ws, int* err,
                    const __grid_constant__ CUtensorMap ta2, const __grid_constant__ CUtensorMap tb2,
                    const __grid_constant__ CUtensorMap tc2, int N2, int K2, int splits2, EpiParams ep2) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  const uint32_t sA = base;
  const uint32_t sB = base + STAGES2 * A2_STAGE_BYTES;
  const uint32_t stg = base + RING2_BYTES;
  const uint32_t bars = stg + STG2_BYTES;
  const uint32_t full0 = bars;
  const uint32_t empty0 = bars + 8 * STAGES2;
  const uint32_t tfull0 = bars + 16 * STAGES2;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;
  const uint32_t holder = drain + 8;
  const uint32_t fix0 = holder + 8;  // 4 x FIX_BOXES stream-K fix-up barriers
  const uint32_t ds_go = fix0 + 8 * 4 * FIX_BOXES;  // DS: the receiver's ring is free (4 warps)
  const uint32_t ds_data0 = ds_go + 8;              // DS: + 8 (4 q + c), chunk c of band q arrived
  volatile uint32_t* holder_ptr = reinterpret_cast<volatile uint32_t*>(smem + (holder - base));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + (holder + 4 - base));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();
  const uint32_t rank = crank & 1u;             // 0: leader of the pair (issues the MMAs), 1: peer
  const uint32_t lead = crank & ~1u;            // cluster rank of this pair's leader
  const uint16_t pair_mask = (uint16_t)(0x3u << lead);
  // the scheduler's unit: the pair (one cluster, or half of a DS cluster)
  const int cluster = (int)(blockIdx.x >> 1);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES2; ++s) {
      mbar_init(full0 + 8 * s, 1);             // the pair leader's producer arrives (+ tx bytes)
      mbar_init(empty0 + 8 * s, 1);            // the pair's MMA commit
    }
    mbar_init(tfull0, 1);
    mbar_init(tfull0 + 8, 1);
    mbar_init(tempty0, 8);  // 4 epilogue warps x 2 CTAs (used in the leader)
    mbar_init(tempty0 + 8, 8);
    mbar_init(drain, 1);
    for (int b = 0; b < 4 * FIX_BOXES; ++b) mbar_init(fix0 + 8 * b, 1);
    mbar_init(ds_go, 4);
    for (int b = 0; b < 16; ++b) mbar_init(ds_data0 + 8 * b, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tma);
    prefetch_tmap(&tmb);
    prefetch_tmap(&tmbh);
    if (FUSE) {
      prefetch_tmap(&ta2);
      prefetch_tmap(&tb2);
    }
  }
  if (warp == 1) tmem_alloc_pair(holder, TMEM2_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the peer's barriers exist before any remote arrive
  tc_fence_after();
  const uint32_t tmem_base = *holder_ptr;
  pdl_wait();  // the previous kernel of the step has completed
  pdl_launch_dependents();
  static_assert(!FUSE || KA2 == 1, "the fused MLP counts its second GEMM's K in 64-column blocks");
  const int num_m_max = (M + 255) / 256;  // (the plan's rows: the layout of the fused counters)
  if (ep.m_dev) M = min(M, *ep.m_dev);  // the step's row count (written by an earlier kernel)
  const int num_m = (M + 255) / 256;
  const int num_n = (N + 255) / 256;
  Sched sc;
  sc.tiles = num_m * num_n;
  sc.ku = (K + BK * KA2 - 1) / (BK * KA2);
  sc.C = gridDim.x / 2;
  sc.splits = splits;
  sc.streamk = streamk;
  sc.halves = halves;
  sc.ds = DS ? 1 : 0;
  sc.fuse = FUSE ? 1 : 0;
  const int num_n2 = FUSE ? (N2 + 255) / 256 : 0;
  sc.tiles2 = num_m * num_n2;
  sc.ku2 = FUSE ? K2 / BK : 0;
  sc.splits2 = FUSE ? splits2 : 1;
  // fused-MLP counters (see above)
  int* const f_ord = flags;
  int* const f_dep = FUSE ? flags + (size_t)num_m_max * num_n2 * 2 : nullptr;
  int* const f_pass = FUSE ? f_dep + (size_t)num_m_max * splits2 : nullptr;
  // item tile -> (m block, n block), M-fastest
  auto tile_mn = [&](int t, int& m_blk, int& n_blk) {
    m_blk = t % num_m;
    n_blk = t / num_m;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer (both CTAs)
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      Item it;
      for (int idx = 0; ok && next_item(idx, sc, cluster, it); ++idx) {
        int m_blk, n_blk;
        tile_mn(it.t, m_blk, n_blk);
        const int kb0 = it.ku0 * KA2, kb1 = it.ku1 * KA2;
        // this CTA's half of the weight rows of the item: 128 rows of a whole tile, or 64
        // of a half-width piece (SwiGLU: the gate rows in the leader, the matching up rows
        // in the peer, as for whole tiles)
        const bool hw = it.width != 256;
        const int wrow = n_blk * 256 +
                         (!hw ? (int)rank * 128
                              : (EPI == EPI_SWIGLU ? (int)rank * 128 + it.piece * 64 : it.piece * 128 + (int)rank * 64));
        const CUtensorMap* tw_map = hw ? &tmbh : &tmb;
        const CUtensorMap* ta_map = &tma;
        if (FUSE && it.g == 1) {
          // the second GEMM reads act columns [ku0 * 64, ku1 * 64) of rows m_blk: wait until
          // the first GEMM's tiles writing them (act columns 128 n .. 128 n + 127 from tile n,
          // both CTAs of its pair) have stored them
          ta_map = &ta2;
          tw_map = &tb2;
          const int need = 2 * ((it.ku1 + 1) / 2 - it.ku0 / 2);
          int* dep = f_dep + m_blk * splits2 + it.sp;
          if (!wait_flag_geq(dep, need, abort_flag)) {
            ok = false;
            break;
          }
          fence_proxy_async_global();  // the act stores (acquired) before this CTA's TMA loads
          // the last of the pair CTAs that wait on this counter resets it for the next launch
          if (atomicAdd(f_pass + m_blk * splits2 + it.sp, 1) == 2 * num_n2 - 1) {
            atomicExch(dep, 0);
            atomicExch(f_pass + m_blk * splits2 + it.sp, 0);
          }
        }
        const uint32_t stage_tx = 2u * (uint32_t)(hw ? A2_STAGE_BYTES + B2_STAGE_BYTES / 2 : STAGE2_BYTES);
        for (int kb = kb0; kb < kb1; kb += KA2) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t full_leader = mapa_shared(full0 + 8 * stage, lead);
          if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * stage, stage_tx);
          for (int a = 0; a < KA2; ++a) {
            tma_load_2d_pair(sA + stage * A2_STAGE_BYTES + a * A_STAGE_BYTES, ta_map, (kb + a) * BK,
                             m_blk * 256 + (int)rank * 128, full_leader);
            tma_load_2d_pair(sB + stage * B2_STAGE_BYTES + a * B2_BLOCK_BYTES, tw_map, (kb + a) * BK, wrow,
                             full_leader);
          }
          if (++stage == STAGES2) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ------------------------------------------------ MMA issuer (leader CTA only)
      constexpr uint32_t idesc_full = make_idesc(256, 256);
      constexpr uint32_t idesc_half = make_idesc(256, 128);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      Item it;
      for (int idx = 0; ok && next_item(idx, sc, cluster, it); ++idx) {
        const int kb0 = it.ku0 * KA2, kb1 = it.ku1 * KA2;
        const uint32_t idesc = it.width == 256 ? idesc_full : idesc_half;
        const int ab = idx & 1;
        const uint32_t aph = (uint32_t)(idx >> 1) & 1u;
        if (!mbar_wait(tempty0 + 8 * ab, aph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * 256);
        for (int kb = kb0; kb < kb1; kb += KA2) {
          if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          // (no tcgen05 fence here: the stage was written by TMA, whose completion the
          // mbarrier itself publishes to the tensor core's async proxy)
#pragma unroll
          for (int a = 0; a < KA2; ++a) {
            const uint64_t da = sw128_desc(sA + stage * A2_STAGE_BYTES + a * A_STAGE_BYTES);
            const uint64_t db = sw128_desc(sB + stage * B2_STAGE_BYTES + a * B2_BLOCK_BYTES);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)
              umma_bf16_pair(d_tmem, da + 2 * k, db + 2 * k, idesc, (kb > kb0 || a > 0 || k > 0) ? 1u : 0u);
          }
          umma_commit_pair(empty0 + 8 * stage, pair_mask);
          if (++stage == STAGES2) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair(tfull0 + 8 * ab, pair_mask);
      }
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
      }
      umma_commit_pair(drain, (uint16_t)(1u << lead));
      volatile int no_abort = 0;
      mbar_wait(drain, 0, &no_abort);
    }
  } else {
    // ------------------------------------------------ epilogue warps 2..5 (both CTAs)
    const int q = warp & 3;                 // TMEM lane quarter = 32-row band of this warp
    const int et = (warp - 2) * 32 + lane;  // 0..127
    const int row_local = q * 32 + lane;
    Stage o;
    o.box0 = stg + (uint32_t)(q * 2 * BOX_BYTES);
    o.lane = lane;
    o.n = 0;
    Item it;
    for (int idx = 0; next_item(idx, sc, cluster, it); ++idx) {
      const int ab = idx & 1;
      const uint32_t aph = (uint32_t)(idx >> 1) & 1u;
      if (!mbar_wait(tfull0 + 8 * ab, aph, abort_flag)) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
        break;
      }
      tc_fence_after();
      int m_blk, n_blk;
      tile_mn(it.t, m_blk, n_blk);
      const int t = m_blk + num_m * n_blk;  // the tile's id for counters and partials
      const int row = m_blk * 256 + (int)rank * 128 + row_local;
      o.row0 = m_blk * 256 + (int)rank * 128 + q * 32;
      o.live = o.row0 < M;
      Src s;
      s.taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * 256);
      s.row = row_local;
      if (it.kind == IT_PLAIN) {
        epilogue_pair<EPI>(s, o, &tmc, &tmv, &tmk, row, n_blk, M, N, ep, it.piece, it.width);
        if (FUSE) {
          // publish the tile's act columns to the second GEMM's items that read them: once
          // this CTA's stores have completed, one arrival per split range they fall in
          o.drain();
          epilogue_bar();
          if (et == 0) {
            __threadfence();
            const int kb_lo = 2 * n_blk, kb_hi = 2 * n_blk + 1;  // its act columns in 64-column K blocks
            const int s_lo = ((kb_lo + 1) * splits2 - 1) / sc.ku2, s_hi = ((kb_hi + 1) * splits2 - 1) / sc.ku2;
            atomicAdd(f_dep + m_blk * splits2 + s_lo, 1);
            if (s_hi != s_lo) atomicAdd(f_dep + m_blk * splits2 + s_hi, 1);
          }
        }
      } else if (FUSE && it.g == 1) {
        // the second GEMM's split it.sp of tile (m_blk, n_blk), added to the residual stream
        // after split it.sp - 1 (a per-tile counter, reset by the last split)
        const int sp = it.sp;
        int* flag = f_ord + (m_blk + num_m * n_blk) * 2 + rank;
        if (et == 0 && !wait_flag_geq(flag, sp, abort_flag)) {
          *abort_flag = 1;
          report_error(err, DERR_WAIT_TIMEOUT);
        }
        epilogue_bar();
        if (!*abort_flag) epilogue_pair<EPI_RESID_F32>(s, o, &tc2, &tmv, &tmk, row, n_blk, M, N2, ep2);
        o.drain();
        epilogue_bar();
        if (et == 0) {
          __threadfence();
          atomicExch(flag, sp + 1 == splits2 ? 0 : sp + 1);
        }
      } else if (it.kind == IT_DS_RECV || it.kind == IT_DS_SEND) {
        // The two K halves of a left-over tile meet half way: the lower-K pair finalises
        // columns [0, 128) of the tile, the upper-K pair columns [128, 256).  Each pair's
        // MMAs are done (tfull), so its operand ring is free: it writes the other pair's
        // 128 columns of its own accumulator there and, once the other pair's ring is free,
        // one bulk copy per (band, 64-column chunk) moves them into the same place of the
        // other pair's ring; then its epilogue adds the received half to its own (lower +
        // upper: one addition, the same value either way round) over its 128 columns,
        // waiting for each received chunk when it first reads it.
        const int mine = it.kind == IT_DS_SEND ? 1 : 0;  // the 128-column piece finalised here
        const uint32_t partner = crank ^ 2u;
        if (lane == 0) {
          for (int c = 0; c < 2; ++c) mbar_arrive_expect_tx(ds_data0 + 8 * (4 * q + 2 * mine + c), DS_BLOCK_BYTES);
          mbar_arrive_cluster(mapa_shared(ds_go, partner));
        }
        __syncwarp();
        bool go = false;
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          const int chunk = 2 * (1 - mine) + c;  // a chunk of the other pair's piece
          const uint32_t blk = sA + (uint32_t)((4 * q + chunk) * DS_BLOCK_BYTES);
          const uint32_t own = blk + (uint32_t)(lane * DS_ROW_BYTES);
#pragma unroll 1
          for (int h = 0; h < 2; ++h) {
            uint32_t r[32];
            tmem_ld32(s.taddr + 64 * chunk + 32 * h, r);
            tmem_ld_wait();
#pragma unroll
            for (int k = 0; k < 8; ++k)
              st_shared_v4(own + (uint32_t)((32 * h + 4 * k) * 4), r[4 * k], r[4 * k + 1], r[4 * k + 2], r[4 * k + 3]);
          }
          fence_proxy_async_smem();  // the rows are read by the bulk copy (async proxy)
          __syncwarp();
          if (!go) {
            if (!mbar_wait_acq_cluster(ds_go, 0, abort_flag)) {
              *abort_flag = 1;
              report_error(err, DERR_WAIT_TIMEOUT);
            }
            go = true;
            __syncwarp();
          }
          if (lane == 0 && !*abort_flag) {
            bulk_copy_to_cluster(mapa_shared(blk, partner), blk, DS_BLOCK_BYTES,
                                 mapa_shared(ds_data0 + 8 * (4 * q + chunk), partner));
            bulk_commit();
          }
        }
        // this pair's piece: TMEM columns and received chunks from 128 * mine on
        s.taddr += (uint32_t)(128 * mine);
        s.dpart = sA + (uint32_t)(2 * mine * 32 * DS_ROW_BYTES);
        s.dbar = ds_data0 + 8 * (4 * q + 2 * mine);
        s.dready = 0;
        s.dabort = abort_flag;
        s.derr = err;
        if (!*abort_flag) epilogue_pair<EPI>(s, o, &tmc, &tmv, &tmk, row, n_blk, M, N, ep, mine, 128);
        // every chunk has landed before this CTA may leave (one the epilogue skipped too),
        // and the other pair has read this CTA's rows (the ring is not touched again)
        for (int c = 0; c < 2; ++c) ds_chunk_ready(s, c);
        if (lane == 0) bulk_wait_read<0>();
        __syncwarp();
      } else if (it.kind == IT_SPLIT) {
        const int sp = it.sp;
        int* flag = flags + t * 2 + rank;
        if constexpr (EPI == EPI_RESID_F32) {
          if (et == 0 && !wait_flag_geq(flag, sp, abort_flag)) {
            *abort_flag = 1;
            report_error(err, DERR_WAIT_TIMEOUT);
          }
          epilogue_bar();
          if (!*abort_flag) epilogue_pair<EPI>(s, o, &tmc, &tmv, &tmk, row, n_blk, M, N, ep);
          o.drain();
          epilogue_bar();
          if (et == 0) {
            __threadfence();
            atomicExch(flag, sp + 1 == splits ? 0 : sp + 1);
          }
        } else {
          const int S1 = splits - 1;
          if (sp < S1) {
            store_partial_pair(s, o, &tmw, ((t * S1 + sp) * 2 + (int)rank) * 128 + q * 32);
            o.drain();
            epilogue_bar();
            if (et == 0) {
              __threadfence();
              atomicAdd(flag, 1);
            }
          } else {
            if (et == 0 && !wait_flag_geq(flag, S1, abort_flag)) {
              *abort_flag = 1;
              report_error(err, DERR_WAIT_TIMEOUT);
            }
            epilogue_bar();
            __threadfence();
            s.part = ws + ((size_t)t * S1 * 2 + rank) * 128 * 256;
            s.part_stride = (size_t)2 * 128 * 256;
            s.nparts = S1;
            if (!*abort_flag) epilogue_pair<EPI>(s, o, &tmc, &tmv, &tmk, row, n_blk, M, N, ep);
            epilogue_bar();
            if (et == 0) atomicExch(flag, 0);
          }
        }
      } else {
        // stream-K segment of left-over tile it.rel
        int* flag = flags + it.rel * 2 + rank;
        const int y_slot0 = ((it.rel * ws_slots) * 2 + (int)rank) * 128 + q * 32;
        if (it.kind == IT_PART) {
          store_partial_pair(s, o, &tmw, y_slot0 + it.slot * 256);
          o.drain();
          epilogue_bar();
          if (et == 0) {
            __threadfence();
            atomicAdd(flag, 1);
          }
        } else {
          if (et == 0 && it.slot > 0 && !wait_flag_geq(flag, it.slot, abort_flag)) {
            *abort_flag = 1;
            report_error(err, DERR_WAIT_TIMEOUT);
          }
          epilogue_bar();
          if (it.slot > 0 && !*abort_flag) {
            const uint32_t tsum = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)((ab ^ 1) * 256);
            if (fixup_to_tmem(&tmw, y_slot0, 256, it.slot, base + (uint32_t)(q * (RING2_BYTES / 4)),
                              fix0 + (uint32_t)(q * 8 * FIX_BOXES), tsum, lane, abort_flag, err)) {
              s.has_sum = true;
              s.tsum = tsum;
            }
          }
          if (!*abort_flag) epilogue_pair<EPI>(s, o, &tmc, &tmv, &tmk, row, n_blk, M, N, ep);
          epilogue_bar();
          if (et == 0) atomicExch(flag, 0);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(tempty0 + 8 * ab, lead));
    }
    if (lane == 0) bulk_wait_read<0>();  // the staging boxes outlive every store reading them
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  __syncwarp();
  cluster_sync_all();  // no CTA leaves while its pair may still touch its smem or TMEM
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM2_COLS);
  }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool encode_kmajor(CUtensorMap* tm, const void* ptr, int rows, int k, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)k, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)k * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Row-major [rows][cols] output / workspace seen in boxes of 32 rows x 128 bytes with
// 128-byte swizzle (the pair epilogue's staging layout).
bool encode_rows(CUtensorMap* tm, void* ptr, CUtensorMapDataType dt, int esize, long rows, long cols, long ld) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * esize};
  cuuint32_t box[2] = {(cuuint32_t)(128 / esize), 32};
  cuuint32_t es[2] = {1, 1};
  return fn(tm, dt, 2, ptr, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int EPI>
cudaError_t launch_t(const GemmPlan& p, int* err, cudaStream_t stream) {
  static bool attr_set = false;
  auto kern = gemm_tc_kernel<BN, EPI>;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)Cfg<BN>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  return launch_pdl(kern, p.grid, NUM_THREADS, Cfg<BN>::SMEM, stream, p.ta, p.tb, p.M, p.N, p.K, p.ep, err);
}

template <int EPI, bool DS = false, bool FUSE = false>
cudaError_t launch_t2(const GemmPlan& p, int* err, cudaStream_t stream) {
  static bool attr_set = false;
  auto kern = gemm_tc2_kernel<EPI, DS, FUSE>;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM2);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = SMEM2;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = DS ? 4 : 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, p.ta, p.tb, p.tbh, p.tc, p.tw, p.tv, p.tk, p.M, p.N, p.K, p.ep, p.splits,
                            p.streamk, p.halves, p.ws_slots, p.flags, p.ws, err, p.ta2, p.tb2, p.tc2, p.N2, p.K2,
                            p.splits2, p.ep2);
}

// Clusters of four CTA-pair CTAs that can be resident at once (0 if unknown).
int cluster4_max() {
  static int n = -1;
  if (n < 0) {
    auto kern = gemm_tc2_kernel<EPI_BF16, true>;
    n = 0;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM2) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(4);
      cfg.blockDim = dim3(NUM_THREADS);
      cfg.dynamicSmemBytes = SMEM2;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 4;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int c = 0;
      if (cudaOccupancyMaxActiveClusters(&c, kern, &cfg) == cudaSuccess) n = c;
    }
    cudaGetLastError();  // a failed query leaves no sticky error
  }
  return n;
}

double wave_efficiency(long tiles, int sms) {
  const long waves = (tiles + sms - 1) / sms;
  return (double)tiles / (double)(waves * sms);
}

}  // namespace

int gemm_lmhead_blocks(int vocab) { return (vocab + 255) / 256; }

bool encode_tmap(CUtensorMap* tm, CUtensorMapDataType dt, int rank, void* ptr, const uint64_t* dims,
                 const uint64_t* strides, const uint32_t* box, CUtensorMapSwizzle swizzle) {
  auto fn = encode_fn();
  if (!fn || rank < 1 || rank > 5) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i + 1 < rank) st[i] = strides[i];
  }
  return fn(tm, dt, rank, ptr, d, st, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t gemm_plan(GemmPlan* plan, const void* A, int M, int K, const void* W, int N, int epi,
                      const EpiParams& ep, int num_sms, int tile, const char** why) {
  *why = nullptr;
  if (M <= 0 || N <= 0 || K <= 0 || K % BK != 0 || (epi != EPI_LMHEAD && N % 32 != 0)) {
    *why = "gemm: need M, N, K > 0, K % 64 == 0 and (except for the LM head) N % 32 == 0";
    return cudaErrorInvalidValue;
  }
  if ((reinterpret_cast<uintptr_t>(A) & 15) || (reinterpret_cast<uintptr_t>(W) & 15)) {
    *why = "gemm: operands must be 16-byte aligned";
    return cudaErrorInvalidValue;
  }
  // Tile choice (measured on the LLaDA-8B step's shapes): the CTA-pair tile keeps the
  // tensor pipe busiest and is used whenever M spans more than one 128-row tile; a
  // residual GEMM whose pair tiles fill less than 3/4 of the GPU and whose K is long
  // splits K in two (ordered adds into the residual stream); small M uses one-CTA tiles,
  // 256 or 128 wide by wave fill.  Stream-K (left-over tiles cut into K segments, fp32
  // partials summed in K order in TMEM) is available on request: every partial costs a
  // 256 KB store and reload per tile, and at ~55 GB/s of stores per SM when all SMs store
  // at once that outweighs the balance it buys on these shapes.
  const bool pair_forced = (tile & 0xff) == kTilePair;
  const bool sk_forced = pair_forced && (tile & kTileStreamK);
  int bn = pair_forced ? kTilePair : (tile & 0xff), cg = 1, splits = 1, streamk = 0;
  const int forced_splits = pair_forced ? ((tile >> 8) & 0xff) : 0;
  const long nkb = (K + BK - 1) / BK;
  const long m1 = (M + BM - 1) / BM;
  const bool wide_only = (epi == EPI_SWIGLU || epi == EPI_LMHEAD);
  const int pairs = num_sms / 2;
  const long units = (K + BK * KA2 - 1) / (BK * KA2);
  const long pair_tiles = (long)((M + 255) / 256) * ((N + 255) / 256);
  const long left = pairs > 0 ? pair_tiles % pairs : 0;
  const int split_auto = (epi == EPI_RESID_F32 && 4 * pair_tiles < 3L * pairs && nkb >= 128) ? 2 : 1;
  if (pair_forced && pairs < 1) {
    *why = "gemm: the CTA-pair tile needs two SMs";
    return cudaErrorInvalidValue;
  }
  if (bn == kTilePair) {
    bn = 256;
    cg = 2;
    if (sk_forced) {
      // forced_splits here counts segments per left-over tile (0: all pairs share them)
      const long csk = forced_splits == 0 ? pairs : std::min<long>(pairs, (long)forced_splits * left);
      if (forced_splits == 1 || left == 0 || left * units < csk) {
        *why = "gemm: stream-K needs a partial last round and at least one K block per sharing pair";
        return cudaErrorInvalidValue;
      }
      streamk = (int)csk;
    } else {
      splits = forced_splits > 0 ? forced_splits : split_auto;
    }
  } else if (bn == 0) {
    if (M > BM && pairs >= 1) {
      bn = 256;
      cg = 2;
      splits = split_auto;
    } else if (wide_only) {
      bn = 256;
    } else {
      const double e256 = wave_efficiency(m1 * ((N + 255) / 256), num_sms);
      const double e128 = 0.9 * wave_efficiency(m1 * ((N + 127) / 128), num_sms);
      bn = (e256 >= e128) ? 256 : 128;
    }
  }
  if (splits < 1 || splits > nkb) {
    *why = "gemm: split count must be in [1, K/64]";
    return cudaErrorInvalidValue;
  }
  if ((epi == EPI_SWIGLU || epi == EPI_LMHEAD) && bn != 256) {
    *why = "gemm: SwiGLU and LM-head epilogues need 256-column tiles";
    return cudaErrorInvalidValue;
  }
  if (bn != 128 && bn != 256) {
    *why = "gemm: tile width must be 128 or 256";
    return cudaErrorInvalidValue;
  }
  if (epi == EPI_SWIGLU && N % 256 != 0) {
    *why = "gemm: SwiGLU needs 2*ffn a multiple of 256";
    return cudaErrorInvalidValue;
  }
  if (epi == EPI_QKV_ROPE && (ep.rope_cols % bn != 0 || bn % ep.head_dim != 0 ||
                              (ep.head_dim != 64 && ep.head_dim != 128))) {
    *why = "gemm: RoPE epilogue needs tile-aligned q|k columns and head_dim 64/128";
    return cudaErrorInvalidValue;
  }
  plan->M = M;
  plan->N = N;
  plan->K = K;
  plan->fuse = 0;
  plan->N2 = plan->K2 = 0;
  plan->splits2 = 1;
  memset(&plan->ta2, 0, sizeof(plan->ta2));
  memset(&plan->tb2, 0, sizeof(plan->tb2));
  memset(&plan->tc2, 0, sizeof(plan->tc2));
  plan->bn = bn;
  plan->cg = cg;
  plan->epi = epi;
  plan->ep = ep;
  if (epi == EPI_LMHEAD) plan->ep.vocab = N;
  // Half-width tail (on request, kTileHalves): whole tiles in full rounds, then each
  // tile of a partial last round as two 256 x 128 pieces on two pairs, with no partial
  // sums to combine (each output is still one MMA chain over all of K, so results are
  // bit-identical to whole tiles).  Measured, a piece takes as long per K block as a
  // whole tile: the six-stage operand ring, not the tensor core, sets the pace of a
  // K block (about 1.7 us of load latency under full load over six 32 KB stages), so the
  // planner does not pick it.
  int halves = 0;
  if (cg == 2 && pair_forced && (tile & kTileHalves)) {
    if (streamk != 0 || epi == EPI_LMHEAD || forced_splits > 1) {
      *why = "gemm: half-width tail tiles exclude stream-K, K splits and the LM-head epilogue";
      return cudaErrorInvalidValue;
    }
    halves = 1;
    splits = 1;
  }
  // each CTA loads 128 rows of A; of W a one-CTA tile loads bn rows, a pair CTA 128
  if (!encode_kmajor(&plan->ta, A, M, K, BM) ||
      !encode_kmajor(&plan->tb, W, N, K, cg == 2 ? 128 : bn) ||
      (cg == 2 && !encode_kmajor(&plan->tbh, W, N, K, 64))) {
    *why = "gemm: cuTensorMapEncodeTiled failed";
    return cudaErrorInvalidValue;
  }
  plan->splits = splits;
  plan->streamk = streamk;
  plan->halves = halves;
  plan->ws_slots = 0;
  plan->flags_needed = 0;
  plan->ws_needed = 0;
  plan->flags = nullptr;
  plan->ws = nullptr;
  memset(&plan->tc, 0, sizeof(plan->tc));
  memset(&plan->tw, 0, sizeof(plan->tw));
  memset(&plan->tv, 0, sizeof(plan->tv));
  memset(&plan->tk, 0, sizeof(plan->tk));
  plan->ep.vt_heads = 0;
  plan->ep.k_store = 0;
  if (cg == 2 && epi != EPI_LMHEAD) {
    const bool f32 = (epi == EPI_RESID_F32);
    const int es = f32 ? 4 : 2;
    const long cols = (epi == EPI_SWIGLU) ? N / 2 : N;
    if ((reinterpret_cast<uintptr_t>(ep.out) & 15) || ((long)ep.ldo * es) % 16 != 0 || ep.ldo < cols) {
      *why = "gemm: the output must be 16-byte aligned with a row pitch of a multiple of 16 bytes";
      return cudaErrorInvalidValue;
    }
    if (!encode_rows(&plan->tc, ep.out, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, es,
                     M, cols, ep.ldo)) {
      *why = "gemm: cuTensorMapEncodeTiled failed (output)";
      return cudaErrorInvalidValue;
    }
  }
  // DSMEM split (kTileDsmem, or chosen by the planner): four-CTA clusters; whole tiles in
  // full rounds over all pairs, then each left-over tile split by K over the two pairs of
  // one cluster, the upper half's fp32 sum written straight into the lower pair's idle
  // operand ring (distributed shared memory, no global partials) and added there before
  // the epilogue.  The last round then costs about half a tile.
  int ds = 0, ds_clusters = 0;
  if (cg == 2) {
    const bool ds_forced = pair_forced && (tile & kTileDsmem);
    const bool ds_ok = streamk == 0 && halves == 0 && epi != EPI_LMHEAD && units >= 2 &&
                       (ds_forced ? forced_splits <= 1 : true);
    const int cl4 = ds_ok ? std::min(num_sms / 4, cluster4_max()) : 0;
    long full = 0, rest = 0;
    if (cl4 >= 1) {
      full = pair_tiles / (2L * cl4);
      rest = pair_tiles % (2L * cl4);
    }
    const bool fits = cl4 >= 1 && rest <= cl4;
    if (ds_forced && !fits) {
      *why = "gemm: the DSMEM split needs four-CTA clusters, no other schedule, K >= 128 and at most one "
             "left-over tile per cluster";
      return cudaErrorInvalidValue;
    }
    if (fits) {
      const double c_plain = (double)((pair_tiles + pairs - 1) / pairs);
      const double c_ds = (double)full + (rest ? 0.56 : 0.0);
      const double c_split = splits > 1 ? 0.5 * (double)((pair_tiles * splits + pairs - 1) / pairs) + 0.15 : 1e9;
      const char* env = getenv("DCL_GEMM_DS");
      const bool allowed = !(env && env[0] == '0');
      // (the planner's own choice: tile 0, or a bare pair tile with no other flag or split)
      const bool auto_sched = tile == 0 || tile == kTilePair;
      if (ds_forced || (allowed && auto_sched && rest > 0 && c_ds < c_plain - 0.05 && c_ds < c_split)) {
        ds = 1;
        splits = 1;
        ds_clusters = full > 0 ? cl4 : (int)rest;
        if (ds_clusters < 1) ds_clusters = 1;
      }
    }
  }
  plan->ds = ds;
  if (ds) plan->splits = 1;
  if (cg == 2) {
    plan->n_tiles = (int)pair_tiles;
    // stream-K: all pairs when there are plain rounds, else only the sharing ones (the
    // kernel derives the round stride from the grid)
    const long items = streamk  ? (pair_tiles >= pairs ? pairs : streamk)
                       : halves ? (pair_tiles >= pairs ? pairs : std::min<long>(pairs, 2 * pair_tiles))
                                : pair_tiles * splits;
    plan->grid = 2 * (int)(items < pairs ? items : pairs);
    if (ds) plan->grid = 4 * ds_clusters;
    plan->smem = SMEM2;
    if (splits > 1) {
      plan->flags_needed = (size_t)plan->n_tiles * 2;
      if (epi != EPI_RESID_F32) plan->ws_needed = (size_t)(splits - 1) * plan->n_tiles * 2 * 256 * 128;
    }
    if (streamk) {
      // left-over tile r's K units [r*U, (r+1)*U) are owned by pairs
      // owner(r*U) .. owner((r+1)*U - 1), owner(u) = ((u + 1) * Csk - 1) / (R * U); all
      // but the last write a partial slot
      const long RU = left * units, csk = streamk;
      long slots = 1;
      for (long r = 0; r < left; ++r) {
        const long c0 = ((r * units + 1) * csk - 1) / RU;
        const long c1 = (((r + 1) * units) * csk - 1) / RU;
        slots = (c1 - c0) > slots ? (c1 - c0) : slots;
      }
      plan->ws_slots = (int)slots;
      plan->flags_needed = (size_t)left * 2;
      plan->ws_needed = (size_t)left * slots * 2 * 256 * 128;
    }
  } else {
    plan->n_tiles = ((M + BM - 1) / BM) * ((N + bn - 1) / bn);
    plan->grid = plan->n_tiles < num_sms ? plan->n_tiles : num_sms;
    plan->smem = (bn == 256) ? Cfg<256>::SMEM : Cfg<128>::SMEM;
  }
  return cudaSuccess;
}

cudaError_t gemm_plan_mlp(GemmPlan* plan, const void* xn, int M, int d, const void* Wgu, int F,
                          const EpiParams& ep_act, const void* Wdown, const EpiParams& ep_res, int num_sms,
                          const char** why) {
  *why = nullptr;
  if (F % 128 != 0 || d % 256 != 0 || M <= 0) {
    *why = "fused MLP: needs F a multiple of 128 and d a multiple of 256";
    return cudaErrorInvalidValue;
  }
  // the gate/up part: CTA-pair tiles, unsplit, in plain rounds
  cudaError_t e = gemm_plan(plan, xn, M, d, Wgu, 2 * F, EPI_SWIGLU, ep_act, num_sms, kTilePair | (1 << 8), why);
  if (e != cudaSuccess) return e;
  if (plan->cg != 2 || plan->ds || plan->splits != 1 || plan->streamk || plan->halves) {
    *why = "fused MLP: the gate/up plan is not a plain CTA-pair plan";
    return cudaErrorInvalidValue;
  }
  if ((reinterpret_cast<uintptr_t>(ep_res.out) & 15) || (reinterpret_cast<uintptr_t>(Wdown) & 15) ||
      ep_res.ldo < d || (ep_res.ldo * 4) % 16) {
    *why = "fused MLP: the residual stream and the down weights must be 16-byte aligned";
    return cudaErrorInvalidValue;
  }
  if (!encode_kmajor(&plan->ta2, ep_act.out, M, F, BM) || !encode_kmajor(&plan->tb2, Wdown, d, F, 128) ||
      !encode_rows(&plan->tc2, ep_res.out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, M, d, ep_res.ldo)) {
    *why = "fused MLP: cuTensorMapEncodeTiled failed";
    return cudaErrorInvalidValue;
  }
  plan->fuse = 1;
  plan->N2 = d;
  plan->K2 = F;
  plan->ep2 = ep_res;
  // the down projection split along K into items as long as a gate/up tile (its K)
  const int ku1 = d / BK, ku2 = F / BK;
  int s2 = (ku2 + ku1 / 2) / ku1;
  s2 = s2 < 1 ? 1 : (s2 > ku2 ? ku2 : s2);
  plan->splits2 = s2;
  const long num_m = (M + 255) / 256, num_n2 = d / 256;
  plan->flags_needed = (size_t)(num_m * num_n2 * 2 + 2 * num_m * s2);
  plan->ws_needed = 0;
  const int pairs = num_sms / 2;
  const long items = num_m * (2L * F / 256) + num_m * num_n2 * s2;
  plan->grid = 2 * (int)(items < pairs ? items : pairs);
  return cudaSuccess;
}

bool gemm_fuse_kv(GemmPlan* p, void* kbuf, void* vt, int batch, int T, int H, int G, int hd, int Tp) {
  if (p->cg != 2 || p->epi != EPI_QKV_ROPE || T % 32 != 0 || p->ep.rope_cols % 256 != 0 || (H * hd) % 256 != 0 ||
      (reinterpret_cast<uintptr_t>(vt) & 15) || (reinterpret_cast<uintptr_t>(kbuf) & 15) || Tp % 8 != 0)
    return false;
  CUtensorMap tv, tk;
  {
    const uint64_t dims[3] = {(uint64_t)T, (uint64_t)hd, (uint64_t)batch * G};
    const uint64_t strides[2] = {(uint64_t)Tp * 2, (uint64_t)hd * Tp * 2};
    const uint32_t box[3] = {32, 64, 1};
    if (!encode_tmap(&tv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, vt, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_NONE))
      return false;
  }
  {
    const uint64_t cols = (uint64_t)G * hd;
    const uint64_t dims[3] = {cols, (uint64_t)T, (uint64_t)batch};
    const uint64_t strides[2] = {cols * 2, (uint64_t)T * cols * 2};
    const uint32_t box[3] = {64, 32, 1};
    if (!encode_tmap(&tk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, kbuf, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
      return false;
  }
  p->tv = tv;
  p->tk = tk;
  p->ep.vt_heads = G;
  p->ep.k_store = 1;
  p->ep.k_col0 = H * hd;
  return true;
}

cudaError_t gemm_bind_scratch(GemmPlan* p, int* flags, float* ws) {
  p->flags = flags;
  p->ws = ws;
  if (p->cg == 2 && p->ws_needed) {
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 15)) return cudaErrorInvalidValue;
    if (!encode_rows(&p->tw, ws, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, (long)(p->ws_needed / 256), 256, 256))
      return cudaErrorInvalidValue;
  }
  return cudaSuccess;
}

// Fault-handling self-test: one thread waits, through the same bounded helpers the
// pipelines use, on something nothing will ever signal - a fresh mbarrier (which = 0) or
// a zero counter in global memory (which = 1) - gives up after the wait limit, records
// DERR_WAIT_TIMEOUT and returns, leaving the context usable.
__global__ void wait_selftest_kernel(int which, const int* flag, int* err) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  bool ok;
  if (which == 0) {
    const uint32_t b = smem_u32(&bar);
    mbar_init(b, 1);
    fence_mbar_init();
    ok = mbar_wait(b, 0, &abort_flag);  // phase 0 completes only after an arrival
  } else {
    ok = wait_flag_geq(flag, 1, &abort_flag);
  }
  if (!ok) report_error(err, DERR_WAIT_TIMEOUT);
}

cudaError_t wait_selftest_launch(int which, const int* flag, int* err, cudaStream_t stream) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(which, flag, err);
  return cudaGetLastError();
}

cudaError_t gemm_launch(const GemmPlan& p, int* err, cudaStream_t stream) {
  if ((p.flags_needed && !p.flags) || (p.ws_needed && !p.ws)) return cudaErrorInvalidValue;
  if (p.fuse) return p.cg == 2 && p.epi == EPI_SWIGLU ? launch_t2<EPI_SWIGLU, false, true>(p, err, stream)
                                                      : cudaErrorInvalidValue;
  if (p.cg == 2 && p.ds) {
    switch (p.epi) {
      case EPI_BF16: return launch_t2<EPI_BF16, true>(p, err, stream);
      case EPI_RESID_F32: return launch_t2<EPI_RESID_F32, true>(p, err, stream);
      case EPI_QKV_ROPE: return launch_t2<EPI_QKV_ROPE, true>(p, err, stream);
      case EPI_SWIGLU: return launch_t2<EPI_SWIGLU, true>(p, err, stream);
    }
    return cudaErrorInvalidValue;
  }
  if (p.cg == 2) {
    switch (p.epi) {
      case EPI_BF16: return launch_t2<EPI_BF16, false>(p, err, stream);
      case EPI_RESID_F32: return launch_t2<EPI_RESID_F32, false>(p, err, stream);
      case EPI_QKV_ROPE: return launch_t2<EPI_QKV_ROPE, false>(p, err, stream);
      case EPI_SWIGLU: return launch_t2<EPI_SWIGLU, false>(p, err, stream);
      case EPI_LMHEAD: return launch_t2<EPI_LMHEAD, false>(p, err, stream);
    }
    return cudaErrorInvalidValue;
  }
  if (p.bn == 256) {
    switch (p.epi) {
      case EPI_BF16: return launch_t<256, EPI_BF16>(p, err, stream);
      case EPI_RESID_F32: return launch_t<256, EPI_RESID_F32>(p, err, stream);
      case EPI_QKV_ROPE: return launch_t<256, EPI_QKV_ROPE>(p, err, stream);
      case EPI_SWIGLU: return launch_t<256, EPI_SWIGLU>(p, err, stream);
      case EPI_LMHEAD: return launch_t<256, EPI_LMHEAD>(p, err, stream);
    }
  } else {
    switch (p.epi) {
      case EPI_BF16: return launch_t<128, EPI_BF16>(p, err, stream);
      case EPI_RESID_F32: return launch_t<128, EPI_RESID_F32>(p, err, stream);
      case EPI_QKV_ROPE: return launch_t<128, EPI_QKV_ROPE>(p, err, stream);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace dcl
