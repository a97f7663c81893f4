// Non-causal (bidirectional) attention of the denoise step's forward: every position
// attends to every position of its sequence, drafts and masks included (App. B.2:
// the dLLMs use bidirectional attention; Sec. 3.3: drafts act as right-side context).
//
//   out[t, h, :] = softmax_j(q[t,h,:] . k[j,g(h),:] / sqrt(hd)) v[j,g(h),:],  j < T
//
// Flash-style single pass with an online softmax (fp32 statistics), bf16 tensor-core
// MMAs (mma.sync m16n8k16), one CTA per (64 queries, head, sequence), 4 warps x 16
// query rows, 64-key K/V tiles double-buffered through cp.async into XOR-swizzled
// shared memory.  GQA: query head h reads kv head h / (H/G).
#include "common.cuh"

namespace dcl {
namespace {

constexpr int BQ = 64;
constexpr int BKV = 64;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, int src_bytes) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// element offset of 16-byte chunk c of row r in a [rows][HD] tile (chunks XOR-swizzled by row)
template <int HD>
__device__ __forceinline__ int soff(int r, int c) {
  return r * HD + ((c ^ (r & 7)) << 3);
}

template <int HD>
__device__ __forceinline__ void load_tile(__nv_bfloat16* s, const __nv_bfloat16* g, int ld, int r0,
                                          int T) {
  constexpr int CH = HD / 8;
  for (int i = threadIdx.x; i < BKV * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const int t = r0 + r;
    const int tc = t < T ? t : T - 1;  // in-bounds address; zero-filled when t >= T
    cp_async16(s + soff<HD>(r, c), g + (size_t)tc * ld + c * 8, t < T ? 16 : 0);
  }
}

template <int HD>
__global__ void __launch_bounds__(128) attn_kernel(const __nv_bfloat16* __restrict__ qkv,
                                                   __nv_bfloat16* __restrict__ out, int T, int H,
                                                   int G, float scale_log2) {
  constexpr int KS = HD / 16;  // k-steps over the head dimension
  constexpr int NT = BKV / 8;  // n8 tiles of scores per key tile
  constexpr int DT = HD / 8;   // n8 tiles of the output
  extern __shared__ uint4 smem4[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem4);
  __nv_bfloat16* sK = sQ + BQ * HD;
  __nv_bfloat16* sV = sK + 2 * BKV * HD;

  const int q0 = blockIdx.x * BQ, h = blockIdx.y, b = blockIdx.z;
  const int g = h / (H / G);
  const int ld = (H + 2 * G) * HD;
  const __nv_bfloat16* base = qkv + (size_t)b * T * ld;
  const __nv_bfloat16* Qg = base + h * HD;
  const __nv_bfloat16* Kg = base + (H + g) * HD;
  const __nv_bfloat16* Vg = base + (H + G + g) * HD;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nkv = (T + BKV - 1) / BKV;

  load_tile<HD>(sQ, Qg, ld, q0, T);
  load_tile<HD>(sK, Kg, ld, 0, T);
  load_tile<HD>(sV, Vg, ld, 0, T);
  cp_async_commit();

  uint32_t qf[KS][4];
  float o[DT][4];
#pragma unroll
  for (int i = 0; i < DT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

  for (int j = 0; j < nkv; ++j) {
    if (j + 1 < nkv) {
      const int nb = (j + 1) & 1;
      load_tile<HD>(sK + nb * BKV * HD, Kg, ld, (j + 1) * BKV, T);
      load_tile<HD>(sV + nb * BKV * HD, Vg, ld, (j + 1) * BKV, T);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int r = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        ldsm_x4(qf[ks], sQ + soff<HD>(r, ks * 2 + (lane >> 4)));
      }
    }
    const __nv_bfloat16* cK = sK + (j & 1) * BKV * HD;
    const __nv_bfloat16* cV = sV + (j & 1) * BKV * HD;

    // S = Q K^T for this warp's 16 rows x 64 keys
    float s[NT][4];
#pragma unroll
    for (int i = 0; i < NT; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int np = 0; np < NT / 2; ++np) {
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        uint32_t kb[4];
        const int r = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        ldsm_x4(kb, cK + soff<HD>(r, ks * 2 + ((lane >> 3) & 1)));
        mma_bf16(s[2 * np], qf[ks], kb[0], kb[1]);
        mma_bf16(s[2 * np + 1], qf[ks], kb[2], kb[3]);
      }
    }
    // scale to log2 units, mask keys beyond the sequence, online softmax
    const int kbase = j * BKV + (lane & 3) * 2;
    float mx[2] = {mrow[0], mrow[1]};
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kbase + nt * 8 + (e & 1);
        s[nt][e] = key < T ? s[nt][e] * scale_log2 : -INFINITY;
        mx[e >> 1] = fmaxf(mx[e >> 1], s[nt][e]);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float alpha = exp2f(mrow[r] - mx[r]);
      lrow[r] *= alpha;
#pragma unroll
      for (int i = 0; i < DT; ++i) {
        o[i][2 * r] *= alpha;
        o[i][2 * r + 1] *= alpha;
      }
      mrow[r] = mx[r];
    }
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        s[nt][e] = exp2f(s[nt][e] - mrow[e >> 1]);
        lrow[e >> 1] += s[nt][e];
      }
    }
    // O += P V with P split into bf16 hi + lo parts (P = hi + lo to ~2^-17 relative): a
    // single bf16 rounding of P would be amplified ~sqrt(T) when attention is diffuse
    // and its output is an average of nearly cancelling value vectors.
#pragma unroll
    for (int kk = 0; kk < BKV / 16; ++kk) {
      uint32_t ph[4], pl[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float* src = s[2 * kk + (e >> 1)] + 2 * (e & 1);
        const __nv_bfloat162 hi = __floats2bfloat162_rn(src[0], src[1]);
        const float2 hf = __bfloat1622float2(hi);
        const __nv_bfloat162 lo = __floats2bfloat162_rn(src[0] - hf.x, src[1] - hf.y);
        ph[e] = *reinterpret_cast<const uint32_t*>(&hi);
        pl[e] = *reinterpret_cast<const uint32_t*>(&lo);
      }
#pragma unroll
      for (int dp = 0; dp < DT / 2; ++dp) {
        uint32_t vb[4];
        const int r = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        ldsm_x4_t(vb, cV + soff<HD>(r, dp * 2 + (lane >> 4)));
        mma_bf16(o[2 * dp], ph, vb[0], vb[1]);
        mma_bf16(o[2 * dp + 1], ph, vb[2], vb[3]);
        mma_bf16(o[2 * dp], pl, vb[0], vb[1]);
        mma_bf16(o[2 * dp + 1], pl, vb[2], vb[3]);
      }
    }
    __syncthreads();
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    lrow[r] = 1.f / lrow[r];
  }
  const int ldo = H * HD;
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int t = q0 + warp * 16 + (lane >> 2) + r * 8;
    if (t < T) {
      uint32_t* dst = reinterpret_cast<uint32_t*>(out + ((size_t)b * T + t) * ldo + h * HD +
                                                  (lane & 3) * 2);
#pragma unroll
      for (int i = 0; i < DT; ++i)
        dst[i * 4] = pack_bf16x2(o[i][2 * r] * lrow[r], o[i][2 * r + 1] * lrow[r]);
    }
  }
}

template <int HD>
cudaError_t launch_hd(const __nv_bfloat16* qkv, __nv_bfloat16* out, int batch, int T, int H, int G,
                      cudaStream_t stream) {
  constexpr size_t smem = (size_t)5 * BQ * HD * sizeof(__nv_bfloat16);
  static bool attr = false;
  if (!attr) {
    cudaError_t e =
        cudaFuncSetAttribute(attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  dim3 grid((T + BQ - 1) / BQ, H, batch);
  const float scale_log2 = kLog2e / sqrtf((float)HD);
  attn_kernel<HD><<<grid, 128, smem, stream>>>(qkv, out, T, H, G, scale_log2);
  return cudaGetLastError();
}

}  // namespace

cudaError_t attention_launch(const __nv_bfloat16* qkv, __nv_bfloat16* out, int batch, int T, int H,
                             int G, int hd, cudaStream_t stream) {
  if (batch <= 0 || T <= 0 || G <= 0 || H % G != 0) return cudaErrorInvalidValue;
  if (hd == 128) return launch_hd<128>(qkv, out, batch, T, H, G, stream);
  if (hd == 64) return launch_hd<64>(qkv, out, batch, T, H, G, stream);
  return cudaErrorInvalidValue;
}

}  // namespace dcl
