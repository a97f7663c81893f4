// Non-causal attention of the bidirectional forward (Eq. 2 runs one full pass in which
// every position attends to every position of its sequence), on the tcgen05 tensor
// cores of sm_103a.
//
// One CTA = 128 query rows of one (sequence, head); the key axis is walked once, in
// blocks of 128: S_j = Q K_j^T into TMEM (double-buffered), then per row a running
// maximum m, P_j = exp2(S_j * log2(e)/sqrt(hd) - m) with the row sum l kept in fp32, P_j
// written to shared memory in fp16 (11 significant bits; P <= 2^8), and O += P_j V_j in
// TMEM with V^T held in fp16 (the bf16 values of v, which fp16 holds exactly).  m moves
// only when a block's maximum exceeds it by more than 8 (P stays below 2^8); l and O are
// then scaled by the same factor, so O / l is unchanged.  O / l leaves through TMA.
//
// Roles (320 threads): warp 0 lane 0 TMA producer (Q once, then K / V^T blocks through a
// 4-stage ring in the order the MMAs consume them); warp 1 allocates TMEM and its lane 0
// issues the MMAs; warps 2..9 run the softmax and the epilogue, two warps per 32-row
// band (TMEM lane quarter), each on one 64-column half of every S block: the block
// maxima and the final sums of the two halves are combined through shared memory.  P is double-buffered so
// that the softmax of block j + 1 overlaps the P V MMAs of block j.  V enters as V^T (a
// K-major operand, kv contiguous, fp16), written by the QKV GEMM's epilogue or by
// v_transpose_kernel from the q|k|v buffer.
// Every wait is bounded (DERR_WAIT_TIMEOUT).
#include "common.cuh"
#include "tc_ptx.cuh"

namespace dcl {
namespace {

constexpr int AT_THREADS = 320;
constexpr int AT_SOFTMAX = 8;  // softmax warps (2 .. 9)
constexpr int AT_STAGES = 4;
constexpr int AT_BOX = 128 * 128;  // one 128-row x 128-byte swizzle box

template <int HD>
struct AttnCfg {
  static constexpr int KB = HD / 64;                   // 64-wide boxes along hd
  static constexpr int Q_BYTES = 128 * HD * 2;         // Q tile [128][HD]
  static constexpr int STAGE_BYTES = 128 * HD * 2;     // K block [128][HD] or V^T block [HD][128]
  static constexpr int VBOX = HD * 128;                // one V^T box: [HD rows][64 kv]
  static constexpr int P_BYTES = 2 * 2 * AT_BOX;       // 2 buffers of P (fp16), [128][128] each
  static constexpr int BARS = 256;
  static constexpr int RED = 2 * 128 * 4;              // per-half row maxima / sums [2][128]
  static constexpr size_t SMEM = 1024 + (size_t)Q_BYTES + AT_STAGES * STAGE_BYTES + P_BYTES + BARS + RED;
  static constexpr uint32_t TMEM_COLS = 512;           // S double buffer (2 x 128) + O (HD)
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

// vt[(b*G + g)*hd + d][t] = v of token t, kv head g, component d (row pitch Tp, zero pad),
// in fp16 (the bf16 values, held exactly).  A block moves a 64-token x 64-channel tile
// with 16-byte loads and stores.
__global__ void __launch_bounds__(256) v_transpose_kernel(const __nv_bfloat16* __restrict__ qkv,
                                                          __half* __restrict__ vt, int T, int Tp, int cols,
                                                          int v0, int ghd) {
  __shared__ __half tile[64][72];  // [channel][token], rows padded by 16 bytes
  pdl_wait();
  pdl_launch_dependents();
  const int t0 = blockIdx.x * 64, c0 = blockIdx.y * 64, b = blockIdx.z;
  for (int i = threadIdx.x; i < 64 * 8; i += 256) {
    const int r = i >> 3, cv = (i & 7) * 8;  // token row, first channel of the vector
    const int t = t0 + r;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (t < T && c0 + cv < ghd)
      v = *reinterpret_cast<const uint4*>(qkv + ((size_t)b * T + t) * cols + v0 + c0 + cv);
    const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&v);
#pragma unroll
    for (int k = 0; k < 8; ++k) tile[cv + k][r] = __float2half_rn(__bfloat162float(e[k]));
  }
  __syncthreads();
  for (int i = threadIdx.x; i < 64 * 8; i += 256) {
    const int c = i >> 3, tv = (i & 7) * 8;  // channel row, first token of the vector
    if (c0 + c < ghd && t0 + tv < Tp)
      *reinterpret_cast<uint4*>(vt + ((size_t)b * ghd + c0 + c) * Tp + t0 + tv) =
          *reinterpret_cast<const uint4*>(&tile[c][tv]);
  }
}

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const __grid_constant__ CUtensorMap to, int T, int H,
                   int G, int kcol0, const int* __restrict__ seq_off, const int* __restrict__ seq_len, int* err) {
  using C = AttnCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  const uint32_t sQ = base;
  const uint32_t sKV = sQ + C::Q_BYTES;
  const uint32_t sP = sKV + AT_STAGES * C::STAGE_BYTES;  // per buffer: two 64-key boxes of P
  const uint32_t bars = sP + C::P_BYTES;
  const uint32_t q_full = bars;
  const uint32_t kv_full0 = bars + 8;                   // + 8 s
  const uint32_t kv_empty0 = kv_full0 + 8 * AT_STAGES;  // + 8 s
  const uint32_t s_full0 = kv_empty0 + 8 * AT_STAGES;   // + 8 b
  const uint32_t s_empty0 = s_full0 + 16;               // + 8 b
  const uint32_t p_full0 = s_empty0 + 16;  // + 8 buffer
  const uint32_t p_empty0 = p_full0 + 16;  // + 8 buffer
  const uint32_t o_full = p_empty0 + 16;
  const uint32_t drain = o_full + 8;
  const uint32_t holder = drain + 8;
  volatile uint32_t* holder_ptr = reinterpret_cast<volatile uint32_t*>(smem + (holder - base));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + (holder + 4 - base));
  float* red = reinterpret_cast<float*>(smem + (bars + C::BARS - base));  // [2][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // grid (head, sequence, query tile): the query tile is the slowest index, so that the
  // CTAs with work come first in dispatch order
  const int h = blockIdx.x, b = blockIdx.y, qt = blockIdx.z;
  const int g = h / (H / G);
  const int nb = (T + 127) / 128;

  // set-up first (it reads nothing that earlier kernels write), so that under programmatic
  // dependent launch it overlaps the tail of the kernel before
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < AT_STAGES; ++s) {
      mbar_init(kv_full0 + 8 * s, 1);
      mbar_init(kv_empty0 + 8 * s, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full0 + 8 * i, 1);
      mbar_init(s_empty0 + 8 * i, AT_SOFTMAX);  // the softmax warps
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(p_full0 + 8 * i, AT_SOFTMAX);
      mbar_init(p_empty0 + 8 * i, 1);
    }
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tq);
    prefetch_tmap(&tk);
    prefetch_tmap(&tv);
    prefetch_tmap(&to);
  }
  if (warp == 1) tmem_alloc(holder, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *holder_ptr;

  pdl_wait();  // the previous kernels of the step (the row plan among them) have completed
  pdl_launch_dependents();
  // the query rows of sequence b are rows [off, off + len) of q and of the output; a tile
  // past them has nothing to do and leaves at once (uniform over the CTA)
  const int q_off = seq_off ? seq_off[b] : b * T;
  const int q_len = seq_len ? seq_len[b] : T;
  if (qt * 128 >= q_len) {
    if (warp == 1) tmem_dealloc(tmem, C::TMEM_COLS);
    return;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      bool ok = true;
      int stage = 0;
      uint32_t phase = 0;
      long issued = 0;
      mbar_arrive_expect_tx(q_full, C::Q_BYTES);
      for (int bx = 0; bx < C::KB; ++bx) tma_load_2d(sQ + bx * AT_BOX, &tq, h * HD + bx * 64, q_off + qt * 128, q_full);
      // consumption order: K_0, K_1, then per j: K_{j+2}, V_j (K only while j + 2 < nb)
      const int n_loads = 2 * nb;
      const int head = nb < 2 ? nb : 2, npairs = nb > 2 ? nb - 2 : 0;
      for (int u = 0; u < n_loads && ok; ++u) {
        bool is_v;
        int j;
        if (u < head) {
          is_v = false, j = u;
        } else {
          const int r = u - head;
          if (r < 2 * npairs) {
            is_v = (r & 1) != 0;
            j = (r >> 1) + (is_v ? 0 : 2);
          } else {
            is_v = true;
            j = npairs + (r - 2 * npairs);
          }
        }
        if (!mbar_wait(kv_empty0 + 8 * stage, phase ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t dst = sKV + stage * C::STAGE_BYTES, bar = kv_full0 + 8 * stage;
        mbar_arrive_expect_tx(bar, C::STAGE_BYTES);
        if (!is_v) {
          for (int bx = 0; bx < C::KB; ++bx)
            tma_load_3d(dst + bx * AT_BOX, &tk, kcol0 + g * HD + bx * 64, j * 128, b, bar);
        } else {
          for (int bx = 0; bx < 2; ++bx) tma_load_3d(dst + bx * C::VBOX, &tv, j * 128 + bx * 64, 0, b * G + g, bar);
        }
        ++issued;
        if (++stage == AT_STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
        // wait (bounded) for the copies this thread issued before leaving
        volatile int no_abort = 0;
        mbar_wait(q_full, 0, &no_abort);
        for (int s = 0; s < AT_STAGES && s < issued; ++s) {
          const long arms = (issued - 1 - s) / AT_STAGES + 1;
          mbar_wait(kv_full0 + 8 * s, (uint32_t)((arms - 1) & 1), &no_abort);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t idesc_s = make_idesc(128, 128);
      constexpr uint32_t idesc_o = make_idesc_f16(128, HD);  // fp16 P and V
      bool ok = mbar_wait(q_full, 0, abort_flag);
      int stage = 0;
      uint32_t phase = 0;
      int si = 0;  // S-buffer uses so far
      auto take = [&](uint32_t& st_addr) -> bool {
        if (!mbar_wait(kv_full0 + 8 * stage, phase, abort_flag)) return false;
        st_addr = sKV + stage * C::STAGE_BYTES;
        return true;
      };
      auto release = [&]() {
        umma_commit(kv_empty0 + 8 * stage);
        if (++stage == AT_STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      };
      auto issue_s = [&]() -> bool {  // S[si & 1] = Q K^T with the K block at the ring head
        uint32_t kaddr;
        if (!take(kaddr)) return false;
        const int sb = si & 1;
        if (!mbar_wait(s_empty0 + 8 * sb, (((uint32_t)si >> 1) & 1u) ^ 1u, abort_flag)) return false;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(sb * 128);
#pragma unroll
        for (int k = 0; k < HD / 16; ++k)
          umma_bf16(d, sw128_desc(sQ + (k >> 2) * AT_BOX) + 2 * (k & 3), sw128_desc(kaddr + (k >> 2) * AT_BOX) + 2 * (k & 3),
                    idesc_s, k > 0 ? 1u : 0u);
        release();
        umma_commit(s_full0 + 8 * sb);
        ++si;
        return true;
      };
      auto issue_pv = [&](int j) -> bool {  // O += P_j V_j (fp16 operands)
        uint32_t vaddr;
        if (!take(vaddr)) return false;
        const int pb = j & 1;
        if (!mbar_wait(p_full0 + 8 * pb, ((uint32_t)j >> 1) & 1u, abort_flag)) return false;
        tc_fence_after();
        const uint32_t d = tmem + 256u;
        const uint32_t pbase = sP + (uint32_t)pb * 2 * AT_BOX;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          umma_bf16(d, sw128_desc(pbase + (k >> 2) * AT_BOX) + 2 * (k & 3), sw128_desc(vaddr + (k >> 2) * C::VBOX) + 2 * (k & 3),
                    idesc_o, (j > 0 || k > 0) ? 1u : 0u);
        release();
        umma_commit(p_empty0 + 8 * pb);
        return true;
      };
      if (ok) ok = issue_s();  // S_0, S_1
      if (ok && nb > 1) ok = issue_s();
      for (int j = 0; ok && j < nb; ++j) {  // S_{j+2} (its buffer frees with P_j) before PV_j
        if (j + 2 < nb) ok = issue_s();
        if (ok) ok = issue_pv(j);
      }
      if (ok) umma_commit(o_full);
      if (!ok) {
        *abort_flag = 1;
        report_error(err, DERR_WAIT_TIMEOUT);
      }
      umma_commit(drain);  // every MMA issued here completes before TMEM is released
      volatile int no_abort = 0;
      mbar_wait(drain, 0, &no_abort);
    }
  } else {
    // ------------------------------------------------ softmax + epilogue (warps 2..9)
    const int q = warp & 3;             // TMEM lane quarter = 32-row band
    const int hs = (warp - 2) >> 2;     // which 64-column half of each S block
    const int co = 64 * hs;
    const int r = q * 32 + lane;        // query row within the tile
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    auto softmax_bar = []() { asm volatile("bar.sync 1, %0;" ::"n"(AT_SOFTMAX * 32) : "memory"); };
    const float scale2 = kLog2e * rsqrtf((float)HD);
    // One pass over the key blocks with a running maximum.  Per block: this half's 64
    // columns of S from TMEM, the block's row maximum combined with the partner warp's
    // half through shared memory, then P = exp2(S scale - m) against the running maximum
    // m.  m is raised only when a block's maximum exceeds it by more than 8 (so P <= 2^8,
    // exact in fp32 and in the hi / lo split); l and this warp's half of O are then scaled
    // by 2^(m_old - m_new) once the previous P V product has completed.  O and l carry
    // the same factor, so O / l is the softmax of the exact-maximum form.
    bool ok = true;
    float m = -INFINITY, l = 0.f;
    const uint32_t band_bar_id = 2u + (uint32_t)q;  // the two warps of this 32-row band
    auto band_bar = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(band_bar_id) : "memory"); };
    for (int j = 0; j < nb; ++j) {  // (no early exit: both warps of a band meet at every barrier)
      const int sb = j & 1, pb = j & 1;
      if (ok) ok = mbar_wait(s_full0 + 8 * sb, ((uint32_t)j >> 1) & 1u, abort_flag);
      if (ok && j >= 2) ok = mbar_wait(p_empty0 + 8 * pb, ((uint32_t)(j - 2) >> 1) & 1u, abort_flag);  // PV_{j-2} read it
      ok = __all_sync(0xffffffffu, ok);
      const int valid = T - j * 128 - co;  // live columns of this half
      uint32_t v[2][32];
      float mm = -INFINITY;
      if (ok) {
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 2; ++c) tmem_ld32(tmem + lane_off + (uint32_t)(sb * 128 + co + 32 * c), v[c]);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(s_empty0 + 8 * sb);  // the S buffer is free for S_{j+2}
        if (valid >= 64) {
          // four independent three-input maximum chains over the 64 columns
          float a4[4];
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const uint32_t* w = &v[t >> 1][(t & 1) * 16];
            float acc = f32(w[0]);
#pragma unroll
            for (int e = 1; e < 15; e += 2) acc = max3f(acc, f32(w[e]), f32(w[e + 1]));
            a4[t] = fmaxf(acc, f32(w[15]));
          }
          mm = max3f(a4[0], a4[1], fmaxf(a4[2], a4[3]));
        } else {
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (32 * c + e < valid) mm = fmaxf(mm, f32(v[c][e]));
        }
      }
      red[hs * 128 + r] = mm * scale2;
      band_bar();
      const float mb = fmaxf(red[r], red[128 + r]);
      band_bar();  // both halves read before the next block writes the slots
      if (!ok) continue;
      const bool raise = mb > m + 8.f;  // always at the first block (m = -inf)
      if (j > 0 && __any_sync(0xffffffffu, raise)) {
        // rescale l and this warp's O columns; P V_{j-1} must have completed first
        if (!mbar_wait(p_empty0 + 8 * ((j - 1) & 1), ((uint32_t)(j - 1) >> 1) & 1u, abort_flag)) ok = false;
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) continue;
        tc_fence_after();
        const float f = raise ? ex2_approx(m - mb) : 1.f;
#pragma unroll 1
        for (int c = co; c < HD && c < co + 64; c += 32) {
          uint32_t ov[32];
          tmem_ld32(tmem + lane_off + 256u + (uint32_t)c, ov);
          tmem_ld_wait();
          float o[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = f32(ov[e]) * f;
          tmem_st32(tmem + lane_off + 256u + (uint32_t)c, o);
        }
        tmem_st_wait();
        tc_fence_before();
        l *= f;
      }
      if (raise) m = mb;
      const uint32_t box = sP + (uint32_t)pb * 2 * AT_BOX + (uint32_t)hs * AT_BOX;
      const bool full = valid >= 64;
      // the block's sum of this half, in two packed partial sums (fixed order)
      unsigned long long la = 0ull, lb = 0ull;
      const unsigned long long sc2 = pk2(scale2, scale2), nm2 = pk2(-m, -m);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        // P in fp16 (round to nearest even: 2^-12 relative, P <= 2^8); l sums the fp32 values
        float pv[32];
        if (full) {  // the exponent arguments two lanes per instruction, no column mask
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float y0, y1;
            upk2(ffma2(pk2(f32(v[c][e]), f32(v[c][e + 1])), sc2, nm2), y0, y1);
            pv[e] = ex2_approx(y0);
            pv[e + 1] = ex2_approx(y1);
          }
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            pv[e] = ex2_approx(fmaf(f32(v[c][e]), scale2, -m));
            if (32 * c + e >= valid) pv[e] = 0.f;
          }
        }
#pragma unroll
        for (int e = 0; e < 32; e += 4) {
          la = fadd2(la, pk2(pv[e], pv[e + 1]));
          lb = fadd2(lb, pk2(pv[e + 2], pv[e + 3]));
        }
        const int k0 = c * 4;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          st_shared_v4(box + swz(r, k0 + k), pack_f16x2(pv[8 * k], pv[8 * k + 1]), pack_f16x2(pv[8 * k + 2], pv[8 * k + 3]),
                       pack_f16x2(pv[8 * k + 4], pv[8 * k + 5]), pack_f16x2(pv[8 * k + 6], pv[8 * k + 7]));
      }
      {
        float a0, a1, b0, b1;
        upk2(la, a0, a1);
        upk2(lb, b0, b1);
        l += (a0 + b0) + (a1 + b1);
      }
      tc_fence_before();
      fence_proxy_async_smem();  // P is read by the tensor cores (async proxy)
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full0 + 8 * pb);
    }
    // the row sum over both halves, half 0 + half 1 (a fixed order)
    red[hs * 128 + r] = l;
    softmax_bar();
    l = red[r] + red[128 + r];
    if (ok) ok = mbar_wait(o_full, 0, abort_flag);
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
      // epilogue: O / l -> bf16 -> TMA store, each warp one 64-column box of its band
      // (staged in the P buffers, free once every PV MMA has completed)
      tc_fence_after();
      const float inv = 1.0f / l;
      const int row0 = qt * 128 + q * 32;
#pragma unroll 1
      for (int c = co; c < HD; c += 128) {
        const uint32_t bx = sP + (uint32_t)((q * 2 + hs) * (32 * 128));
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t v[32];
          tmem_ld32(tmem + lane_off + 256u + (uint32_t)(c + 32 * hh), v);
          tmem_ld_wait();
          float o[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = f32(v[e]) * inv;
#pragma unroll
          for (int k = 0; k < 4; ++k)
            st_shared_v4(bx + swz(lane, 4 * hh + k), pack_bf16x2(o[8 * k], o[8 * k + 1]), pack_bf16x2(o[8 * k + 2], o[8 * k + 3]),
                         pack_bf16x2(o[8 * k + 4], o[8 * k + 5]), pack_bf16x2(o[8 * k + 6], o[8 * k + 7]));
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0 && row0 < q_len) {
          if (seq_off)
            tma_store_2d(&to, bx, h * HD + c, q_off + row0);
          else
            tma_store_3d(&to, bx, h * HD + c, row0, b);
        }
      }
      if (lane == 0) {
        bulk_commit();
        bulk_wait_read<0>();  // the staging boxes were read (the writes complete with the grid)
      }
      __syncwarp();
    }
    if (!ok) {
      *abort_flag = 1;
      report_error(err, DERR_WAIT_TIMEOUT);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int HD>
cudaError_t launch_attn(const AttnPlan& p, int* err, cudaStream_t stream) {
  static bool attr_set = false;
  auto kern = attn_tc_kernel<HD>;
  if (!attr_set) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AttnCfg<HD>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid(p.H, p.batch, (p.T + 127) / 128);
  return launch_pdl(kern, grid, AT_THREADS, AttnCfg<HD>::SMEM, stream, p.tq, p.tk, p.tv, p.to, p.T, p.H, p.G, p.kcol0,
                    p.seq_off, p.seq_len, err);
}

}  // namespace

int attn_vt_pitch(int T) { return (T + 7) & ~7; }

cudaError_t attention_plan(AttnPlan* p, const __nv_bfloat16* qkv, const __nv_bfloat16* kbuf, __half* vt,
                           __nv_bfloat16* out, int batch, int T, int H, int G, int hd, int rows_max,
                           const int* seq_off, const int* seq_len) {
  if (batch <= 0 || T <= 0 || H <= 0 || G <= 0 || H % G || (hd != 64 && hd != 128) || rows_max <= 0)
    return cudaErrorInvalidValue;
  if ((reinterpret_cast<uintptr_t>(qkv) & 15) || (reinterpret_cast<uintptr_t>(vt) & 15) ||
      (reinterpret_cast<uintptr_t>(out) & 15) || (kbuf && (reinterpret_cast<uintptr_t>(kbuf) & 15)))
    return cudaErrorInvalidValue;
  const uint64_t cols = (uint64_t)(H + 2 * G) * hd, ocols = (uint64_t)H * hd, Tp = attn_vt_pitch(T);
  {  // q rows of the step: [rows_max][cols]
    const uint64_t dims[2] = {cols, (uint64_t)rows_max};
    const uint64_t strides[1] = {cols * 2};
    const uint32_t box[2] = {64, 128};
    if (!encode_tmap(&p->tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<__nv_bfloat16*>(qkv), dims, strides, box,
                     CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  {  // keys of every position as [batch][T][kcols]: the key store, or the k columns of q|k|v
    const uint64_t kcols = kbuf ? (uint64_t)G * hd : cols;
    const uint64_t dims[3] = {kcols, (uint64_t)T, (uint64_t)batch};
    const uint64_t strides[2] = {kcols * 2, (uint64_t)T * kcols * 2};
    const uint32_t box[3] = {64, 128, 1};
    if (!encode_tmap(&p->tk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(kbuf ? kbuf : qkv), dims,
                     strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    p->kcol0 = kbuf ? 0 : H * hd;
  }
  {  // v^T as [batch*G][hd][T] (row pitch Tp)
    const uint64_t dims[3] = {(uint64_t)T, (uint64_t)hd, (uint64_t)batch * G};
    const uint64_t strides[2] = {Tp * 2, (uint64_t)hd * Tp * 2};
    const uint32_t box[3] = {64, (uint32_t)hd, 1};
    if (!encode_tmap(&p->tv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, vt, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  if (seq_off) {  // output rows of the step: [rows_max][H*hd] (32-row bands of one sequence)
    const uint64_t dims[2] = {ocols, (uint64_t)rows_max};
    const uint64_t strides[1] = {ocols * 2};
    const uint32_t box[2] = {64, 32};
    if (!encode_tmap(&p->to, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, out, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  } else {  // [batch][T][H*hd]: stores of rows past T are clipped
    const uint64_t dims[3] = {ocols, (uint64_t)T, (uint64_t)batch};
    const uint64_t strides[2] = {ocols * 2, (uint64_t)T * ocols * 2};
    const uint32_t box[3] = {64, 32, 1};
    if (!encode_tmap(&p->to, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, out, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  p->qkv = qkv;
  p->vt = vt;
  p->seq_off = seq_off;
  p->seq_len = seq_len;
  p->batch = batch;
  p->T = T;
  p->H = H;
  p->G = G;
  p->hd = hd;
  return cudaSuccess;
}

cudaError_t attention_transpose_launch(const AttnPlan& p, cudaStream_t stream) {
  const int cols = (p.H + 2 * p.G) * p.hd, ghd = p.G * p.hd;
  dim3 tgrid((attn_vt_pitch(p.T) + 63) / 64, (ghd + 63) / 64, p.batch);
  return launch_pdl(v_transpose_kernel, tgrid, 256, 0, stream, p.qkv, p.vt, p.T, attn_vt_pitch(p.T), cols,
                    (p.H + p.G) * p.hd, ghd);
}

cudaError_t attention_core_launch(const AttnPlan& p, int* err, cudaStream_t stream) {
  return p.hd == 128 ? launch_attn<128>(p, err, stream) : launch_attn<64>(p, err, stream);
}

cudaError_t attention_launch(const AttnPlan& p, int* err, cudaStream_t stream) {
  const cudaError_t e = attention_transpose_launch(p, stream);
  return e != cudaSuccess ? e : attention_core_launch(p, err, stream);
}

}  // namespace dcl
