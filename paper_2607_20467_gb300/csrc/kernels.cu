// Bandwidth- and latency-bound kernels of the denoise step:
//   embed_remask   Eq. remasking (draft invalidation, Sec. 3.3 step (i)) fused with the
//                  embedding gather that starts the forward
//   rmsnorm        fp32 residual stream -> bf16 GEMM operand
//   lmhead_combine per-row merge of the LM-head epilogue partials into the top-1 id,
//                  top-1 probability and top-2 probability of Eq. 2's softmax
//   dcv_commit     Eq. compute_k + commit + Eq. draft_update + advance (Sec. 3.3 steps
//                  (iii)-(iv), Algorithm 1), one warp per sequence
//   accept_*       the same acceptance on caller-provided bf16 logits
//   generate       counter-based synthetic weight generator
#include <math.h>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace dcl {
namespace {

constexpr unsigned kFull = 0xffffffffu;

// ------------------------------------------------------------------ step row plan
// One CTA: per sequence the first computed position (0 under full recompute and on a cache
// refresh, the block-aligned prefix end N + Bk*floor((p-N)/Bk) when the stored keys and
// values are that block's, T for a finished row), the row offsets, and the row tables.
__global__ void __launch_bounds__(1024) row_plan_kernel(RowPlan rp, const int32_t* __restrict__ p, int B, int N,
                                                        int T, int Bk, int cached, int update,
                                                        int32_t* __restrict__ x, int window, int mask_id) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ int lm_off[];  // [B], then the sequences' first computed positions [B]
  int* st_pos = lm_off + B;
  const int M = T - N;
  if (threadIdx.x == 0) {
    int off = 0, lmoff = 0;
    for (int b = 0; b < B; ++b) {
      const int pb = p[b];
      int start, end = T, cap = T;
      if (pb >= T) {
        start = T;
      } else if (!cached) {
        start = 0;
      } else {
        const int pe = N + Bk * ((pb - N) / Bk);
        start = (rp.pe_cache[b] == pe) ? pe : 0;
        if (update) rp.pe_cache[b] = pe;
        if (cached == 2 && start != 0) {  // dual cache between refreshes: the current block
          end = min(pe + Bk, T);
          cap = end - pb;
        }
      }
      rp.seq_off[b] = off;
      rp.seq_len[b] = end - start;
      rp.kcap[b] = cap;
      st_pos[b] = start;
      off += end - start;
      lm_off[b] = lmoff;
      lmoff += max(end - max(start, N), 0);
    }
    rp.counts[0] = off;
    rp.counts[1] = lmoff;
  }
  __syncthreads();
  for (int b = 0; b < B; ++b) {
    const int len = rp.seq_len[b], off = rp.seq_off[b], start = st_pos[b], end = start + len;
    for (int i = threadIdx.x; i < len; i += blockDim.x) {
      rp.row_seq[off + i] = b;
      rp.row_pos[off + i] = start + i;
    }
    if (cached == 2 && window > 0 && p[b] < T) {
      // Eq. remasking over the window positions past the computed rows (the embedding
      // kernel re-masks the computed ones): between refreshes of the dual cache the window
      // runs past the block
      const int pb = p[b], w0 = max(pb, end), w1 = min(pb + window, T);
      for (int t = w0 + threadIdx.x; t < w1; t += blockDim.x) x[(size_t)b * T + t] = mask_id;
    }
    const int s0 = max(start, N);
    for (int i = threadIdx.x; i < end - s0; i += blockDim.x) {
      const int pos = s0 + i;
      rp.lm_src[lm_off[b] + i] = off + (pos - start);
      rp.lm_slot[lm_off[b] + i] = b * M + (pos - N);
    }
  }
}

// ------------------------------------------------------------------ embedding + remask
// Row r of the step (grid: the most rows a step can have) is position row_pos[r] of
// sequence row_seq[r]; rows past the step's count return.
__global__ void embed_remask_kernel(int32_t* __restrict__ x, const int32_t* __restrict__ p, int T,
                                    int window, int mask_id, int vocab,
                                    const __nv_bfloat16* __restrict__ embed, int d,
                                    float* __restrict__ h, int* err, RowPlan rp) {
  pdl_wait();
  pdl_launch_dependents();
  const int row = blockIdx.x;
  if (row >= rp.counts[0]) return;
  const int b = rp.row_seq[row], t = rp.row_pos[row];
  __shared__ int tok_s;
  if (threadIdx.x == 0) {
    const int pb = p[b];
    int tok = x[(size_t)b * T + t];
    if (t >= pb && t - pb < window) {  // x_{p+i} <- MASK for i in [0, L)
      tok = mask_id;
      x[(size_t)b * T + t] = mask_id;
    }
    if (tok < 0 || tok >= vocab) {
      report_error(err, DERR_TOKEN_RANGE);
      tok = mask_id;
    }
    tok_s = tok;
  }
  __syncthreads();
  const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)tok_s * d);
  float4* dst = reinterpret_cast<float4*>(h + (size_t)row * d);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) {
    const uint4 v = __ldg(src + i);
    dst[2 * i] = make_float4(bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y));
    dst[2 * i + 1] = make_float4(bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w));
  }
}

// ------------------------------------------------------------------ RMSNorm
template <int THREADS>
__global__ void __launch_bounds__(THREADS) rmsnorm_kernel(const float* __restrict__ x,
                                                          const __nv_bfloat16* __restrict__ gain,
                                                          __nv_bfloat16* __restrict__ y, int d,
                                                          float eps, const int* __restrict__ rows_dev,
                                                          const int* __restrict__ src) {
  pdl_wait();
  pdl_launch_dependents();
  const int r = blockIdx.x;
  if (rows_dev && r >= *rows_dev) return;
  const int in_row = src ? src[r] : r;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)in_row * d);
  const int n4 = d / 4;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n4; i += THREADS) {
    const float4 v = xr[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  __shared__ float red[THREADS / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(kFull, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < THREADS / 32 ? red[threadIdx.x] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(red[0] / (float)d + eps);
  const uint2* g2 = reinterpret_cast<const uint2*>(gain);
  uint2* y2 = reinterpret_cast<uint2*>(y + (size_t)r * d);
  for (int i = threadIdx.x; i < n4; i += THREADS) {
    const float4 v = xr[i];
    const uint2 g = __ldg(g2 + i);
    y2[i] = make_uint2(pack_bf16x2(v.x * inv * bf16_lo(g.x), v.y * inv * bf16_hi(g.x)),
                       pack_bf16x2(v.z * inv * bf16_lo(g.y), v.w * inv * bf16_hi(g.y)));
  }
}

// Single pass: ROWS rows per CTA, 128 threads per row, each thread keeping its
// VPT float4 of the row in registers between the sum of squares and the scaling.
template <int VPT, int ROWS>
__global__ void __launch_bounds__(128 * ROWS) rmsnorm_reg_kernel(
    const float* __restrict__ x, const __nv_bfloat16* __restrict__ gain, __nv_bfloat16* __restrict__ y,
    int rows, int d, float eps, const int* __restrict__ rows_dev, const int* __restrict__ src) {
  pdl_wait();
  pdl_launch_dependents();
  if (rows_dev) rows = min(rows, *rows_dev);
  const int sub = threadIdx.x >> 7, t = threadIdx.x & 127;
  const int r = blockIdx.x * ROWS + sub;
  const bool live = r < rows;
  const int in_row = live ? (src ? src[r] : r) : 0;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)in_row * d);
  const int n4 = d / 4;
  float4 v[VPT];
  uint2 gv[VPT];  // (the gain, loaded with the row: a load next to each store waited for it)
  const uint2* g2 = reinterpret_cast<const uint2*>(gain);
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int j = t + 128 * i;
    v[i] = (live && j < n4) ? xr[j] : make_float4(0.f, 0.f, 0.f, 0.f);
    gv[i] = (live && j < n4) ? __ldg(g2 + j) : make_uint2(0u, 0u);
  }
#pragma unroll
  for (int i = 0; i < VPT; ++i) ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(kFull, ss, o);
  __shared__ float red[ROWS][4];
  if ((t & 31) == 0) red[sub][t >> 5] = ss;
  __syncthreads();
  const float tot = red[sub][0] + red[sub][1] + red[sub][2] + red[sub][3];
  const float inv = rsqrtf(tot / (float)d + eps);
  if (!live) return;
  uint2* y2 = reinterpret_cast<uint2*>(y + (size_t)r * d);
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int j = t + 128 * i;
    if (j < n4) {
      const uint2 g = gv[i];
      y2[j] = make_uint2(pack_bf16x2(v[i].x * inv * bf16_lo(g.x), v[i].y * inv * bf16_hi(g.x)),
                         pack_bf16x2(v[i].z * inv * bf16_lo(g.y), v[i].w * inv * bf16_hi(g.y)));
    }
  }
}

// ------------------------------------------------------------------ softmax partial merge
// A partial is {max m, sum exp(z - m), argmax id, second largest z, sum exp(z - m) * y}
// over some columns, y = (z - m) log2(e) (the last one gives the entropy:
// H = -sum P ln P = ln 2 * (log2(sum) - u / sum)).
struct Part {  // (aggregate: brace-initialised parts leave u = 0)
  float m, s, t2;
  int id;
  float u;
};

__device__ __forceinline__ void merge(Part& a, const Part& b) {
  if (b.m == -INFINITY) return;
  if (a.m == -INFINITY) {
    a = b;
    return;
  }
  const float m = fmaxf(a.m, b.m);
  const float da = (a.m - m) * kLog2e, db = (b.m - m) * kLog2e;  // <= 0, finite; one is 0
  const float ea = da == 0.f ? 1.f : exp2f(da), eb = db == 0.f ? 1.f : exp2f(db);
  const float s = a.s * ea + b.s * eb;
  // re-based to the new maximum: y' = y + d for every term
  const float u = ea * fmaf(da, a.s, a.u) + eb * fmaf(db, b.s, b.u);
  if (b.m > a.m || (b.m == a.m && b.id < a.id)) {
    a.t2 = fmaxf(b.t2, a.m);
    a.id = b.id;
  } else {
    a.t2 = fmaxf(a.t2, b.m);
  }
  a.m = m;
  a.s = s;
  a.u = u;
}

__device__ __forceinline__ Part shfl_part(const Part& a, int off) {
  Part b;
  b.m = __shfl_xor_sync(kFull, a.m, off);
  b.s = __shfl_xor_sync(kFull, a.s, off);
  b.t2 = __shfl_xor_sync(kFull, a.t2, off);
  b.id = __shfl_xor_sync(kFull, a.id, off);
  b.u = __shfl_xor_sync(kFull, a.u, off);
  return b;
}

__device__ __forceinline__ void write_conf(const Part& a, const ConfOut& o, int r) {
  o.top1[r] = a.id;
  // p1 = exp(max - max) / sum.  The sum holds the max's own term exp(0) = 1, but that
  // term is evaluated as exp2 of a rounding residual and may come out a hair below 1, so
  // the probabilities are clamped to [0, 1] and p2 <= p1.
  const float inv = 1.0f / a.s;
  const float c1 = fminf(inv, 1.0f);
  if (o.p1) o.p1[r] = c1;
  if (o.p2) o.p2[r] = a.t2 == -INFINITY ? 0.f : fminf(exp2f((a.t2 - a.m) * kLog2e) * inv, c1);
  if (o.ent || o.mode) {
    // H = -sum P ln P >= 0 (clamped: a near-certain row can round a hair below 0)
    const float h = fmaxf(kLn2 * (log2f(a.s) - a.u * inv), 0.f);
    if (o.ent) o.ent[r] = h;
    if (o.conf) o.conf[r] = o.mode ? expf(-h) : c1;
  } else if (o.conf && o.conf != o.p1) {
    o.conf[r] = c1;
  }
}

// LM row `row` (of *rows_dev) is written to slot slot[row] of top1 / p1 / p2.
// One CTA of COMBINE_THREADS per row: each thread merges a strided share of the row's
// partials, then warps and the CTA merge in a fixed order (deterministic).
constexpr int COMBINE_THREADS = 128;
__global__ void __launch_bounds__(COMBINE_THREADS) lmhead_combine_kernel(
    const float4* __restrict__ part, const float* __restrict__ upart, int rows, int nblk, ConfOut out,
    const int* __restrict__ rows_dev, const int* __restrict__ slot) {
  pdl_wait();
  pdl_launch_dependents();
  const int row = blockIdx.x;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (rows_dev) rows = min(rows, *rows_dev);
  if (row >= rows) return;
  Part a{-INFINITY, 0.f, -INFINITY, 0x7fffffff};
  for (int i = threadIdx.x; i < nblk; i += COMBINE_THREADS) {
    const size_t j = (size_t)row * nblk + i;
    const float4 v = part[j];
    merge(a, Part{v.x, v.y, v.w, __float_as_int(v.z), upart ? upart[j] : 0.f});
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) merge(a, shfl_part(a, o));
  __shared__ Part red[COMBINE_THREADS / 32];
  if (lane == 0) red[w] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    Part t = red[0];
    for (int k = 1; k < COMBINE_THREADS / 32; ++k) merge(t, red[k]);
    write_conf(t, out, slot ? slot[row] : row);
  }
}

// ------------------------------------------------------------------ DCV on one sequence
// xrow / ids / c indexed by absolute position; window [pb, pb + min(L, T - pb)).
// Runs on one full warp.  Returns K (valid on every lane).
__device__ int dcv_row(int32_t* xrow, const int32_t* ids, const float* c, int pb, int T,
                       const DcvParams& prm, int kmax) {
  const int lane = threadIdx.x & 31;
  const int w_eff = min(prm.window, T - pb);
  // Eq. compute_k: K = sum_i prod_{j<=i} 1(c_{p+j} > tau_commit) = length of the leading
  // run of passing positions; each 32-wide chunk is one ballot.
  int K = 0;
  for (int base = 0; base < w_eff; base += 32) {
    const int i = base + lane;
    const bool ok = i < w_eff && c[pb + i] > prm.tau_commit;
    const unsigned bal = __ballot_sync(kFull, ok);
    if (bal == kFull) {
      K += 32;
      continue;
    }
    K += __ffs(~bal) - 1;
    break;
  }
  K = min(min(max(K, prm.min_commit), w_eff), kmax);  // (kmax: the dual cache's block end)
  for (int i = lane; i < K; i += 32) xrow[pb + i] = ids[pb + i];  // commit x[p:p+K]
  // Eq. draft_update over the future region i >= p + L (p before the advance)
  const int lo = pb + prm.window;
  if (!prm.contiguous_drafts) {
    for (int i = lo + lane; i < T; i += 32)
      if (c[i] > prm.tau_draft) xrow[i] = ids[i];
  } else {  // App. E variant: only the unbroken chain starting at p + L
    for (int base = lo; base < T; base += 32) {
      const int i = base + lane;
      const bool ok = i < T && c[i] > prm.tau_draft;
      const unsigned bal = __ballot_sync(kFull, ok);
      const int run = (bal == kFull) ? 32 : __ffs(~bal) - 1;
      if (lane < run) xrow[i] = ids[i];
      if (run < 32) break;
    }
  }
  return K;
}

// ------------------------------------------------------------------ Eq. threshold_pd
// The non-contiguous rule on one row, one full warp: every uncommitted position of
// [lo, hi) with c > tau_commit is committed in the same step (Eq. threshold_pd, applied
// independently per position); when fewer than min_commit pass, the min_commit
// uncommitted positions of highest confidence are committed instead (ties to the lower
// position: round r takes the best position ranked strictly after round r-1's, so nothing
// needs marking).  cmt (committed flags by absolute position) may be NULL: then every
// position of [lo, hi) is uncommitted.  Returns the number committed; *hsum / *hmax get the
// sum and maximum of ent over the committed set (warp-uniform; ent may be NULL).
__device__ int threshold_row(int32_t* xrow, uint8_t* cmt, const int32_t* ids, const float* c, const float* ent,
                             int lo, int hi, const DcvParams& prm, float* hsum, float* hmax) {
  const int lane = threadIdx.x & 31;
  int npass = 0;
  for (int base = lo; base < hi; base += 32) {
    const int i = base + lane;
    const bool ok = i < hi && !(cmt && cmt[i]) && c[i] > prm.tau_commit;
    npass += __popc(__ballot_sync(kFull, ok));
  }
  float hs = 0.f, hm = 0.f;
  int K = 0;
  if (npass >= prm.min_commit) {
    for (int i = lo + lane; i < hi; i += 32) {
      if (!(cmt && cmt[i]) && c[i] > prm.tau_commit) {
        xrow[i] = ids[i];
        if (cmt) cmt[i] = 1;
        if (ent) {
          hs += ent[i];
          hm = fmaxf(hm, ent[i]);
        }
      }
    }
    K = npass;
  } else {
    float pc = INFINITY;  // the previous pick's key (confidence, position)
    int pi = -1;
    for (int r = 0; r < prm.min_commit; ++r) {
      float bc = -INFINITY;
      int bi = 0x7fffffff;
      for (int i = lo + lane; i < hi; i += 32) {
        if (cmt && cmt[i]) continue;
        const float ci = c[i];
        const bool after = ci < pc || (ci == pc && i > pi);  // ranked after the previous pick
        if (after && (ci > bc || (ci == bc && i < bi))) {
          bc = ci;
          bi = i;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float oc = __shfl_xor_sync(kFull, bc, o);
        const int oi = __shfl_xor_sync(kFull, bi, o);
        if (oc > bc || (oc == bc && oi < bi)) {
          bc = oc;
          bi = oi;
        }
      }
      if (bi == 0x7fffffff) break;  // no uncommitted position left in the block
      if (lane == 0) {
        xrow[bi] = ids[bi];
        if (cmt) cmt[bi] = 1;
        if (ent) {
          hs += ent[bi];
          hm = fmaxf(hm, ent[bi]);
        }
      }
      pc = bc;
      pi = bi;
      ++K;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    hs += __shfl_xor_sync(kFull, hs, o);
    hm = fmaxf(hm, __shfl_xor_sync(kFull, hm, o));
  }
  *hsum = hs;
  *hmax = hm;
  __syncwarp();  // this warp's commits (x and flags) are visible to all its lanes
  return K;
}

__global__ void dcv_commit_kernel(int32_t* __restrict__ x, int32_t* __restrict__ p,
                                  int32_t* __restrict__ k_out, int32_t* __restrict__ steps,
                                  const int32_t* __restrict__ ids, const float* __restrict__ c,
                                  const float* __restrict__ ent, float* __restrict__ jpde, int N, int M,
                                  DcvParams prm, int32_t* done_count, uint8_t* __restrict__ cmt,
                                  const int* __restrict__ kcap) {
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.x;
  const int T = N + M;
  const int pb = p[b];
  if (pb >= T) {
    if (threadIdx.x == 0) k_out[b] = 0;
    return;
  }
  if (prm.acceptance == 1) {
    // Eq. threshold_pd in the semi-autoregressive block holding p, then p moves to the
    // leftmost uncommitted position
    const int lo = N + prm.block_len * ((pb - N) / prm.block_len), hi = min(lo + prm.block_len, T);
    uint8_t* crow = cmt + (size_t)b * T;
    float hs, hm;
    const int K = threshold_row(x + (size_t)b * T, crow, ids + (size_t)b * M - N, c + (size_t)b * M - N,
                                ent ? ent + (size_t)b * M - N : nullptr, lo, hi, prm, &hs, &hm);
    int np = T;
    for (int base = pb; base < T; base += 32) {
      const int i = base + (threadIdx.x & 31);
      const unsigned bal = __ballot_sync(kFull, i < T && !crow[i]);
      if (bal) {
        np = base + __ffs(bal) - 1;
        break;
      }
    }
    if (threadIdx.x == 0) {
      if (ent) jpde[b] += K > 1 ? hs - hm : 0.f;
      k_out[b] = K;
      p[b] = np;
      steps[b] += 1;
      if (np >= T) atomicAdd(done_count, 1);
    }
    return;
  }
  // shift the [M]-sized generation arrays so they are indexed by absolute position
  const int K = dcv_row(x + (size_t)b * T, ids + (size_t)b * M - N, c + (size_t)b * M - N, pb, T, prm,
                        kcap ? kcap[b] : T);
  if (ent) {
    // Eq. entropy_bound of the committed set U = [p, p + K): sum_U H - max_U H
    const float* h = ent + (size_t)b * M - N + pb;
    float sum = 0.f, mx = 0.f;
    for (int i = threadIdx.x; i < K; i += 32) {
      sum += h[i];
      mx = fmaxf(mx, h[i]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sum += __shfl_xor_sync(kFull, sum, o);
      mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
    }
    if (threadIdx.x == 0) jpde[b] += K > 1 ? sum - mx : 0.f;
  }
  if (threadIdx.x == 0) {
    k_out[b] = K;
    p[b] = pb + K;
    steps[b] += 1;
    if (pb + K >= T) atomicAdd(done_count, 1);
  }
}

// ------------------------------------------------------------------ block acceptance
// One column into a thread's online partial (columns arrive in increasing order).  ENT
// keeps the entropy sum u (needed only for the entropy confidence).
template <bool ENT>
__device__ __forceinline__ void take1(Part& a, float v, int col) {
  if (v > a.m) {
    const float d = (a.m - v) * kLog2e;  // -inf for the first column
    const float e = exp2f(d);
    if (ENT) a.u = a.s > 0.f ? e * fmaf(d, a.s, a.u) : 0.f;
    a.s = a.s * e + 1.f;
    a.t2 = a.m;
    a.m = v;
    a.id = col;
  } else if (a.m != -INFINITY) {
    if (v > a.t2) a.t2 = v;
    const float y = (v - a.m) * kLog2e;
    const float e = exp2f(y);
    a.s += e;
    if (ENT) a.u = fmaf(e, fmaxf(y, -200.f), a.u);  // e = 0 below -149: the term's limit 0
  }
}

// Eight consecutive columns (one 16-byte vector), without a branch per column: the
// vector's maximum first (a new running maximum rescales s and u once, and takes the
// lowest column holding it as the argmax), then every column adds exp2((z - m) log2 e)
// on the special-function unit.  The argmax's own term is exp2 of the rounding residual
// of the fused multiply-add, within an ulp of 1 (write_conf clamps p1 and p2).  A vector
// holding an infinity takes the exact column-by-column path.
template <bool ENT>
__device__ __forceinline__ void take8(Part& a, const uint4& q, int col) {
  const float v[8] = {bf16_lo(q.x), bf16_hi(q.x), bf16_lo(q.y), bf16_hi(q.y),
                      bf16_lo(q.z), bf16_hi(q.z), bf16_lo(q.w), bf16_hi(q.w)};
  const float cm = fmaxf(max3f(max3f(v[0], v[1], v[2]), max3f(v[3], v[4], v[5]), v[6]), v[7]);
  if (!(fabsf(cm) < INFINITY)) {
#pragma unroll
    for (int k = 0; k < 8; ++k) take1<ENT>(a, v[k], col + k);
    return;
  }
  if (cm > a.m) {
    int k0 = 7;
#pragma unroll
    for (int k = 6; k >= 0; --k) k0 = v[k] == cm ? k : k0;  // lowest column holding the maximum
    float s2 = -INFINITY;  // largest of the other seven
#pragma unroll
    for (int k = 0; k < 8; ++k) s2 = k == k0 ? s2 : fmaxf(s2, v[k]);
    const float d = (a.m - cm) * kLog2e;  // -inf before the first vector
    const float e = exp2f(d);
    if (ENT) a.u = a.s > 0.f ? e * fmaf(d, a.s, a.u) : 0.f;
    a.s *= e;
    a.t2 = fmaxf(a.m, s2);
    a.m = cm;
    a.id = col + k0;
  } else {
    a.t2 = fmaxf(a.t2, cm);
  }
  // y = z log2(e) - m log2(e) and its exp2 for the eight columns, two lanes per
  // instruction; the eight terms are summed as a tree of pairs
  const float ml = a.m * kLog2e;
  const unsigned long long l2 = pk2(kLog2e, kLog2e), nm = pk2(-ml, -ml);
  unsigned long long e2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    float y0, y1;
    upk2(ffma2(pk2(v[2 * k], v[2 * k + 1]), l2, nm), y0, y1);
    const float x0 = ex2_approx(y0), x1 = ex2_approx(y1);
    e2[k] = pk2(x0, x1);
    if (ENT) a.u = fmaf(x1, fmaxf(y1, -200.f), fmaf(x0, fmaxf(y0, -200.f), a.u));
  }
  float s0, s1;
  upk2(fadd2(fadd2(e2[0], e2[1]), fadd2(e2[2], e2[3])), s0, s1);
  a.s += s0 + s1;
}

// One CTA of THREADS per uncommitted position: thread t takes the 16-byte vectors t, t +
// THREADS, ... of the row, ACC_AHEAD of them loaded before any is used (several loads in
// flight per thread: with one, the latency of each load paced the thread).  256 threads
// and at most 32 registers keep eight CTAs, so that ~1200 rows, resident on the 152 SMs at
// once.  CTA a takes the a-th uncommitted position (row by row), so that the CTAs with
// work are the first of the grid and spread evenly over the SMs; the committed positions'
// CTAs, which read nothing, come last (with one CTA per position in place, the live rows
// landed unevenly: 3 on some SMs, 10 on others).
constexpr int ACC_THREADS = 256;
constexpr int ACC_AHEAD = 4;
constexpr int ACC_COMPACT_MAX_B = 256;  // (each CTA scans the rows; larger batches keep one CTA per position in place)
// The a-th uncommitted position of the block (row-major over B rows of P positions, c_b
// committed in row b): its index b * P + i, or -1 if there are fewer (warp-wide call).
__device__ __forceinline__ int nth_uncommitted(const int32_t* committed, int B, int P, int a) {
  const int lane = threadIdx.x & 31;
  for (int b0 = 0; b0 < B; b0 += 32) {
    const int b = b0 + lane;
    const int n = b < B ? P - min(max(committed[b], 0), P) : 0;  // uncommitted positions of row b
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += t;
    }
    const int total = __shfl_sync(kFull, incl, 31);
    if (a < total) {
      const unsigned hit = __ballot_sync(kFull, a < incl);
      const int l = __ffs(hit) - 1;  // the first row whose running count passes a
      const int before = __shfl_sync(kFull, incl - n, l);
      const int nl = __shfl_sync(kFull, n, l);
      return (b0 + l) * P + (P - nl) + (a - before);
    }
    a -= total;
  }
  return -1;
}

template <int THREADS, bool ENT>
__global__ void __launch_bounds__(THREADS, 2048 / THREADS) accept_stats_kernel(
    const __nv_bfloat16* __restrict__ logits, const int32_t* __restrict__ committed, int B, int P, int V,
    int32_t* __restrict__ ids, float* __restrict__ c1, float* __restrict__ c2, int mode) {
  pdl_wait();  // the logits, and the previous call's commit pass that read this scratch
  pdl_launch_dependents();
  int pos = blockIdx.x;  // b * P + i
  if (B <= ACC_COMPACT_MAX_B) {
    __shared__ int pos_s;
    if (threadIdx.x < 32) {
      const int q = nth_uncommitted(committed, B, P, (int)blockIdx.x);
      if (threadIdx.x == 0) pos_s = q;
    }
    __syncthreads();
    pos = pos_s;
    if (pos < 0) return;  // (uniform over the CTA)
  } else if (pos % P < committed[pos / P]) {
    return;  // committed positions are never read
  }
  const __nv_bfloat16* row = logits + (size_t)pos * V;
  Part a{-INFINITY, 0.f, -INFINITY, 0x7fffffff};
  const bool vec = ((reinterpret_cast<uintptr_t>(row) & 15) == 0);
  int done = 0;
  if (vec) {
    const uint4* r4 = reinterpret_cast<const uint4*>(row);
    const int n8 = V / 8;
    int j = threadIdx.x;
    for (; j + (ACC_AHEAD - 1) * THREADS < n8; j += ACC_AHEAD * THREADS) {
      uint4 q[ACC_AHEAD];
#pragma unroll
      for (int t = 0; t < ACC_AHEAD; ++t) q[t] = __ldcs(r4 + j + t * THREADS);
#pragma unroll
      for (int t = 0; t < ACC_AHEAD; ++t) take8<ENT>(a, q[t], (j + t * THREADS) * 8);
    }
    for (; j < n8; j += THREADS) take8<ENT>(a, __ldcs(r4 + j), j * 8);  // streamed once
    done = n8 * 8;
  }
  const unsigned short* r2 = reinterpret_cast<const unsigned short*>(row);
  for (int j = done + threadIdx.x; j < V; j += THREADS) take1<ENT>(a, __uint_as_float((uint32_t)r2[j] << 16), j);
  // a thread's columns arrive in increasing order, so its argmax is its lowest maximal
  // column; merge() breaks ties between threads by the lower id
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) merge(a, shfl_part(a, o));
  __shared__ Part red[THREADS / 32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = a;
  __syncthreads();
  if (threadIdx.x < 32) {
    Part v = threadIdx.x < THREADS / 32 ? red[threadIdx.x] : Part{-INFINITY, 0.f, -INFINITY, 0x7fffffff};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) merge(v, shfl_part(v, o));
    if (threadIdx.x == 0) {
      ConfOut o;
      o.top1 = ids;
      o.p2 = c2;
      o.conf = c1;
      o.mode = mode;
      write_conf(v, o, pos);
    }
  }
}

__global__ void accept_commit_kernel(const int32_t* __restrict__ committed,
                                     const int32_t* __restrict__ ids, const float* __restrict__ c1,
                                     int32_t* __restrict__ x, int32_t* __restrict__ k, int P,
                                     DcvParams prm) {
  pdl_wait();  // the statistics pass
  pdl_launch_dependents();
  const int b = blockIdx.x;
  const int pb = committed[b];
  if (pb >= P || pb < 0) {
    if (threadIdx.x == 0) k[b] = 0;
    return;
  }
  int K;
  if (prm.acceptance == 1) {  // Eq. threshold_pd over the uncommitted rest [c_b, P), no drafts
    float hs, hm;
    K = threshold_row(x + (size_t)b * P, nullptr, ids + (size_t)b * P, c1 + (size_t)b * P, nullptr, pb, P, prm, &hs,
                      &hm);
  } else {
    K = dcv_row(x + (size_t)b * P, ids + (size_t)b * P, c1 + (size_t)b * P, pb, P, prm, P);
  }
  if (threadIdx.x == 0) k[b] = K;
}

// ------------------------------------------------------------------ launch floor
// A kernel that does nothing but the step kernels' dependent-launch handshake: a graph of
// n of them measures the launch cost a step of n launches cannot go below.
__global__ void empty_step_kernel() {
  pdl_wait();
  pdl_launch_dependents();
}

// ------------------------------------------------------------------ weight generator
__device__ __forceinline__ uint64_t splitmix64(uint64_t z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__global__ void generate_kernel(__nv_bfloat16* __restrict__ dst, uint64_t seed, int tid,
                                int64_t start, int64_t count, float scale, float mean,
                                int64_t cols, int blk, int blk_stride, int blk_off) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count; e += stride) {
    const uint64_t idx = (uint64_t)(start + e);
    const uint64_t h = splitmix64((seed << 48) | ((uint64_t)tid << 32) | idx);
    const int s = (int)(h & 0xFFFF) + (int)((h >> 16) & 0xFFFF) + (int)((h >> 32) & 0xFFFF) +
                  (int)(h >> 48);
    float w = __fmul_rn((float)(s - 131070), scale);  // no fused multiply-add: exact IEEE ops
    if (mean != 0.f) w = __fadd_rn(w, mean);
    int64_t o = e;
    if (blk > 0) {
      const int64_t r = (int64_t)idx / cols, cidx = (int64_t)idx % cols;
      o = ((r / blk) * blk_stride + blk_off + r % blk) * cols + cidx;
    }
    dst[o] = __float2bfloat16_rn(w);
  }
}

}  // namespace

// ------------------------------------------------------------------ launchers
cudaError_t row_plan_launch(const RowPlan& rp, const int32_t* p, int batch, int N, int T, int block_len, int cached,
                            int update, int32_t* x, int window, int mask_id, cudaStream_t stream) {
  if (batch <= 0 || batch > 4096 || (cached && block_len <= 0) || cached < 0 || cached > 2 || (cached == 2 && !x))
    return cudaErrorInvalidValue;
  return launch_pdl(row_plan_kernel, 1, 1024, 2 * sizeof(int) * batch, stream, rp, p, batch, N, T, block_len, cached,
                    update, x, window, mask_id);
}

cudaError_t embed_remask_launch(int32_t* x, const int32_t* p, int batch, int T, int window,
                                int mask_id, int vocab, const __nv_bfloat16* embed, int d, float* h,
                                int* err, const RowPlan& rp, cudaStream_t stream) {
  if (d % 8) return cudaErrorInvalidValue;
  return launch_pdl(embed_remask_kernel, batch * T, 128, 0, stream, x, p, T, window, mask_id, vocab, embed, d, h, err,
                    rp);
}

cudaError_t rmsnorm_launch(const float* x, const __nv_bfloat16* gain, __nv_bfloat16* y, int rows, int d,
                           float eps, const int* rows_dev, const int* src, cudaStream_t stream) {
  if (d % 4 || rows <= 0) return cudaErrorInvalidValue;
  const int vpt = (d / 4 + 127) / 128;  // float4 per thread with 128 threads per row
  const int grid2 = (rows + 1) / 2;
  switch (vpt) {
    case 1: return launch_pdl(rmsnorm_reg_kernel<1, 2>, grid2, 256, 0, stream, x, gain, y, rows, d, eps, rows_dev, src);
    case 2: return launch_pdl(rmsnorm_reg_kernel<2, 2>, grid2, 256, 0, stream, x, gain, y, rows, d, eps, rows_dev, src);
    case 4: case 3: return launch_pdl(rmsnorm_reg_kernel<4, 2>, grid2, 256, 0, stream, x, gain, y, rows, d, eps, rows_dev, src);
    case 5: case 6: case 7: case 8:
      return launch_pdl(rmsnorm_reg_kernel<8, 2>, grid2, 256, 0, stream, x, gain, y, rows, d, eps, rows_dev, src);
    default:
      return launch_pdl(rmsnorm_kernel<256>, rows, 256, 0, stream, x, gain, y, d, eps, rows_dev, src);
  }
}

cudaError_t lmhead_combine_launch(const float4* part, const float* upart, int rows, int nblk, const ConfOut& o,
                                  const int* rows_dev, const int* slot, cudaStream_t stream) {
  return launch_pdl(lmhead_combine_kernel, rows, COMBINE_THREADS, 0, stream, part, upart, rows, nblk, o, rows_dev,
                    slot);
}

cudaError_t dcv_commit_launch(int32_t* x, int32_t* p, int32_t* k_out, int32_t* steps,
                              const int32_t* ids, const float* c, const float* ent, float* jpde, int batch,
                              int N, int M, const DcvParams& prm, int32_t* done_count, uint8_t* cmt,
                              const int* kcap, cudaStream_t stream) {
  if (prm.acceptance == 1 && (prm.block_len < 1 || !cmt)) return cudaErrorInvalidValue;
  return launch_pdl(dcv_commit_kernel, batch, 32, 0, stream, x, p, k_out, steps, ids, c, ent, jpde, N, M, prm,
                    done_count, cmt, kcap);
}

cudaError_t accept_stats_launch(const __nv_bfloat16* logits, const int32_t* committed, int B, int P,
                                int V, int32_t* ids, float* c1, float* c2, int mode, cudaStream_t stream) {
  // Both passes are dependent launches: each is scheduled while its predecessor drains and
  // waits for it (pdl_wait) before touching memory.
  if (mode)
    return launch_pdl(accept_stats_kernel<ACC_THREADS, true>, B * P, ACC_THREADS, 0, stream, logits, committed, B, P,
                      V, ids, c1, c2, mode);
  return launch_pdl(accept_stats_kernel<ACC_THREADS, false>, B * P, ACC_THREADS, 0, stream, logits, committed, B, P, V,
                    ids, c1, c2, mode);
}

cudaError_t accept_commit_launch(const int32_t* committed, const int32_t* ids, const float* c1,
                                 int32_t* x, int32_t* k, int B, int P, const DcvParams& prm,
                                 cudaStream_t stream) {
  return launch_pdl(accept_commit_kernel, B, 32, 0, stream, committed, ids, c1, x, k, P, prm);
}

cudaError_t empty_launch(cudaStream_t stream) { return launch_pdl(empty_step_kernel, 1, 32, 0, stream); }

cudaError_t generate_launch(__nv_bfloat16* dst, uint64_t seed, int tid, int64_t start, int64_t count,
                            float std, float mean, int64_t cols, int blk, int blk_stride, int blk_off,
                            cudaStream_t stream) {
  if (count <= 0) return cudaSuccess;
  const double sigma4 = sqrt(4.0 * (65536.0 * 65536.0 - 1.0) / 12.0);
  const float scale = (float)((double)std / sigma4);
  int64_t blocks = (count + 255) / 256;
  if (blocks > 152 * 32) blocks = 152 * 32;
  generate_kernel<<<(int)blocks, 256, 0, stream>>>(dst, seed, tid, start, count, scale, mean, cols, blk,
                                                   blk_stride, blk_off);
  return cudaGetLastError();
}

cudaError_t rope_table_build(float* cos_dev, float* sin_dev, int T, int hd, float theta,
                             cudaStream_t stream) {
  const int half = hd / 2;
  float* hc = nullptr;
  cudaError_t e = cudaMallocHost(&hc, sizeof(float) * 2 * (size_t)T * half);
  if (e != cudaSuccess) return e;
  for (int t = 0; t < T; ++t)
    for (int j = 0; j < half; ++j) {
      const double ang = (double)t * pow((double)theta, -2.0 * j / hd);
      hc[(size_t)j * T + t] = (float)cos(ang);  // [half][T]: positions contiguous
      hc[(size_t)T * half + (size_t)j * T + t] = (float)sin(ang);
    }
  e = cudaMemcpyAsync(cos_dev, hc, sizeof(float) * (size_t)T * half, cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(sin_dev, hc + (size_t)T * half, sizeof(float) * (size_t)T * half,
                        cudaMemcpyHostToDevice, stream);
  cudaError_t s = cudaStreamSynchronize(stream);
  cudaFreeHost(hc);
  return e != cudaSuccess ? e : s;
}

}  // namespace dcl
