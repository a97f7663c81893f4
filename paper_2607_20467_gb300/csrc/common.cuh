// Shared device helpers and the internal (C++) interface between the library's
// translation units.  Nothing here is part of the C ABI (include/dcleap.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dcl {

// ---------------------------------------------------------------- device error word
// Kernels never trap: they record the first fault here and return.  The host reads
// the word at its sync points and turns it into a dcl_status.
enum DevErr : int {
  DERR_NONE = 0,
  DERR_TOKEN_RANGE = 1,     // a token id outside [0, vocab) reached the embedding
  DERR_WAIT_TIMEOUT = 2,    // a bounded wait gave up (GEMM / attention pipeline)
  DERR_BAD_SHAPE = 3,       // a kernel was launched with a shape it does not support
};

__device__ __forceinline__ void report_error(int* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

// ---------------------------------------------------------------- dependent launch
// Every kernel of the step is launched with programmatic stream serialisation: it may
// start (prologue: barriers, TMEM, tensor-map prefetch) while the previous kernel drains,
// and waits in pdl_wait() until that kernel has completed and its writes are visible.
// Every step kernel calls pdl_wait() before it reads or writes global memory, so the
// order of the step is unchanged (and transitively so: no kernel completes before its
// predecessor has).  pdl_launch_dependents() lets the next kernel be scheduled.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------- small helpers
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------- GEMM (gemm_tc.cu)
// out = A[M][K] @ W[N][K]^T on tcgen05 tensor cores, with a fused epilogue.
enum Epilogue : int {
  EPI_BF16 = 0,      // out bf16 [M][ldo]
  EPI_RESID_F32 = 1, // out float [M][ldo] += acc
  EPI_QKV_ROPE = 2,  // out bf16 [M][ldo]; rotate-half RoPE on columns < rope_cols
  EPI_SWIGLU = 3,    // W rows interleaved per 128: gate block then up block; out bf16
                     // [M][ldo] column n = silu(gate_n) * up_n
  EPI_LMHEAD = 4,    // per (row, 256-column block): float4 {max, sum exp(z-max),
                     // argmax id (bits), second largest z}; columns >= vocab ignored
};

struct EpiParams {
  void* out = nullptr;
  int ldo = 0;
  const float* rope_cos = nullptr;  // [head_dim/2][rope_T], positions contiguous
  const float* rope_sin = nullptr;
  int rope_T = 0;                   // positions in the tables (row length)
  int rope_cols = 0;
  int head_dim = 0;
  int seq_T = 1;                    // rows per sequence (position = row % seq_T)
  int vocab = 0;
  int vt_heads = 0;                 // QKV: > 0 writes v transposed (G kv heads) through tv
  int k_store = 0;                  // QKV: 1 writes k (after RoPE) through tk, not to out
  int k_col0 = 0;                   // QKV: first k column (H * head_dim)
  const int* m_dev = nullptr;       // device row count (<= M) of the launch, or NULL
  const int* row_pos = nullptr;     // device position of each row (NULL: row % seq_T)
  const int* row_seq = nullptr;     // device sequence of each row (NULL: row / seq_T)
  float* ent_part = nullptr;        // LM head: [rows][tiles] sum of e * y (entropy partials) or NULL
};

struct GemmPlan {
  CUtensorMap ta, tb;
  CUtensorMap tbh;       // pair tiles: the weight seen in 64-row boxes (half-width pieces)
  CUtensorMap tc;        // pair tiles: the output (bf16 / fp32 boxes of 32 rows x 128 bytes)
  CUtensorMap tw;        // pair tiles with partials: the fp32 workspace [rows][256]
  CUtensorMap tv;        // QKV with ep.vt_heads > 0: v^T boxes [64 channels][32 tokens]
  CUtensorMap tk;        // QKV with ep.k_store: k boxes [32 tokens][64 channels] of [B][T][G*hd]
  int M = 0, N = 0, K = 0;
  int bn = 256;          // output columns per tile
  int cg = 1;            // 1: one CTA per 128 x bn tile; 2: a CTA pair per 256 x 256 tile
  int epi = EPI_BF16;
  EpiParams ep;
  int grid = 0;
  int n_tiles = 0;
  size_t smem = 0;
  int splits = 1;          // split-K factor (pair tiles only)
  int streamk = 0;         // > 0: left-over pair tiles shared out by K over this many pairs
  int halves = 0;          // 1: the left-over pair tiles run as two 256 x 128 pieces
  int ds = 0;              // 1: four-CTA clusters, left-over tiles split by K over two pairs (DSMEM sum)
  int ws_slots = 0;        // stream-K partial slots per left-over tile
  size_t flags_needed = 0; // ints of zero-initialised split counters the launch needs
  size_t ws_needed = 0;    // floats of workspace for split-K partials
  int* flags = nullptr;    // set through gemm_bind_scratch when flags_needed > 0
  float* ws = nullptr;     // set through gemm_bind_scratch when ws_needed > 0
  // fused MLP (gemm_plan_mlp): one persistent launch runs the gate/up tiles (this plan, SwiGLU
  // into ep.out = act) and then the down projection's K-split tiles (act @ Wdown^T added to
  // the residual stream ep2.out), each down item waiting only for the gate/up tiles that
  // produce its K range of act
  int fuse = 0;
  CUtensorMap ta2, tb2, tc2;  // down: act [M][F] (A), Wdown [d][F] (W), residual [M][d] fp32 (out)
  int N2 = 0, K2 = 0, splits2 = 1;
  EpiParams ep2;
};

// Encode the tensor maps and choose the tile / grid.  A is [M][K] bf16 (row pitch K),
// W is [N][K] bf16.  tile: 0 lets the planner choose; 128 or 256 force a one-CTA tile of
// that width; kTilePair forces the CTA-pair 256 x 256 tile, kTilePair | (S << 8) that
// tile with S K splits (S = 0: the planner chooses, S = 1: unsplit),
// kTilePair | kTileStreamK | (S << 8) the pair tile with the stream-K schedule, each
// left-over tile cut into about S K segments (S = 0: shared out over all pairs).
constexpr int kTilePair = 2;
constexpr int kTileStreamK = 1 << 16;
constexpr int kTileHalves = 1 << 18;     // with kTilePair: left-over tiles as two half-width pieces
constexpr int kTileDsmem = 1 << 19;      // with kTilePair: left-over tiles split by K over a cluster's pairs
cudaError_t gemm_plan(GemmPlan* plan, const void* A, int M, int K, const void* W, int N,
                      int epi, const EpiParams& ep, int num_sms, int tile, const char** why);
// The fused MLP of one layer: act = SwiGLU(xn @ Wgu^T) (Wgu [2F][d], gate / up rows
// interleaved per 128; ep_act.out = act [M][F]) and then h += act @ Wdown^T (Wdown [d][F];
// ep_res.out = h, fp32 [M][d]) in one launch of CTA-pair tiles; F a multiple of 128.
cudaError_t gemm_plan_mlp(GemmPlan* plan, const void* xn, int M, int d, const void* Wgu, int F,
                          const EpiParams& ep_act, const void* Wdown, const EpiParams& ep_res, int num_sms,
                          const char** why);
// Attach the zero-initialised counters (>= flags_needed ints) and the workspace
// (>= ws_needed floats, 16-byte aligned) a plan needs; they may be shared by plans that
// run one after another on one stream.
cudaError_t gemm_bind_scratch(GemmPlan* plan, int* flags, float* ws);
// Make a CTA-pair QKV plan write k (after RoPE) into kbuf (bf16 [batch][T][G*hd]) and v
// transposed into vt (bf16 [batch*G][hd][Tp]) instead of the k and v columns of its
// output, the positions / sequences of its rows given by ep.row_pos / ep.row_seq; false
// (plan unchanged) when the shape does not allow it (T a multiple of 32 is needed).
bool gemm_fuse_kv(GemmPlan* plan, void* kbuf, void* vt, int batch, int T, int H, int G, int hd, int Tp);
cudaError_t gemm_launch(const GemmPlan& plan, int* err, cudaStream_t stream);
// Bounded-wait self-test (which = 0: an mbarrier, 1: a global counter; flag = a zero int).
cudaError_t wait_selftest_launch(int which, const int* flag, int* err, cudaStream_t stream);
int gemm_lmhead_blocks(int vocab);  // number of 256-column partial records per row
// cuTensorMapEncodeTiled through the runtime's driver entry point: dims / box in elements
// (innermost first), strides in bytes for dimensions 1 .. rank-1; out-of-range elements
// read as zero.
bool encode_tmap(CUtensorMap* tm, CUtensorMapDataType dt, int rank, void* ptr, const uint64_t* dims,
                 const uint64_t* strides, const uint32_t* box, CUtensorMapSwizzle swizzle);

// ---------------------------------------------------------------- attention (attention_tc.cu)
// softmax(q k^T / sqrt(hd)) v per (sequence, head): the query rows of sequence b are rows
// [seq_off[b], seq_off[b] + seq_len[b]) of qkv (q columns) and of out (NULL tables: b*T and
// T; with tables every seq_len and seq_off is a multiple of 32), its keys and values are
// all T positions: keys from kbuf [batch][T][G*hd] (NULL: the
// k columns of qkv, rows b*T + t), values from vt [batch*G][hd][attn_vt_pitch(T)]
// (v transposed, in fp16 holding the bf16 values exactly: the attention_transpose_launch
// output, or what the QKV epilogue wrote).
struct AttnPlan {
  CUtensorMap tq, tk, tv, to;
  const __nv_bfloat16* qkv = nullptr;
  __half* vt = nullptr;
  const int* seq_off = nullptr;
  const int* seq_len = nullptr;
  int batch = 0, T = 0, H = 0, G = 0, hd = 0, kcol0 = 0;
};
int attn_vt_pitch(int T);
cudaError_t attention_plan(AttnPlan* p, const __nv_bfloat16* qkv, const __nv_bfloat16* kbuf, __half* vt,
                           __nv_bfloat16* out, int batch, int T, int H, int G, int hd, int rows_max,
                           const int* seq_off, const int* seq_len);
cudaError_t attention_launch(const AttnPlan& p, int* err, cudaStream_t stream);  // both kernels
cudaError_t attention_transpose_launch(const AttnPlan& p, cudaStream_t stream);  // v -> vt
cudaError_t attention_core_launch(const AttnPlan& p, int* err, cudaStream_t stream);  // the attention

// ---------------------------------------------------------------- other kernels (kernels.cu)
// The rows a step computes, in order: sequence b contributes positions [start_b, T) at
// rows [seq_off[b], seq_off[b] + seq_len[b]); start_b is 0 under full recompute and on a
// cache refresh, the block-aligned prefix end otherwise, T for a finished sequence.  The
// LM rows are the computed rows at generation positions.  Written on the device at the
// start of every step, read by the step's kernels (the step graph is shape-static).
struct RowPlan {
  int* counts = nullptr;    // [2]: computed rows R, LM rows R_lm
  int* row_seq = nullptr;   // [B*T] sequence of row r
  int* row_pos = nullptr;   // [B*T] position of row r
  int* seq_off = nullptr;   // [B]
  int* seq_len = nullptr;   // [B]
  int* lm_src = nullptr;    // [B*M] computed row of LM row j
  int* lm_slot = nullptr;   // [B*M] b*M + position - N of LM row j
  int* pe_cache = nullptr;  // [B] prefix end the stored keys / values belong to (-1: none)
  int* kcap = nullptr;      // [B] cap on the step's K: the block end - p between refreshes of the
                            // dual cache, T otherwise
};
// cached: 0 every position; 1 the prefix cache (all positions at a refresh, else from the
// block-aligned prefix end to T); 2 the dual cache (as 1, but between refreshes only the
// current block).  update = 0 plans the rows without recording the prefix end (a forward
// that commits nothing, e.g. a debug pass, leaves the next step's refresh decision
// unchanged).
cudaError_t row_plan_launch(const RowPlan& rp, const int32_t* p, int batch, int N, int T, int block_len,
                            int cached, int update, int32_t* x, int window, int mask_id, cudaStream_t stream);
cudaError_t embed_remask_launch(int32_t* x, const int32_t* p, int batch, int T, int window,
                                int mask_id, int vocab, const __nv_bfloat16* embed, int d,
                                float* h, int* err, const RowPlan& rp, cudaStream_t stream);
// y row r = normalised x row src[r] (src NULL: r), for r < min(rows, *rows_dev).
cudaError_t rmsnorm_launch(const float* x, const __nv_bfloat16* gain, __nv_bfloat16* y, int rows,
                           int d, float eps, const int* rows_dev, const int* src, cudaStream_t stream);
// Per-position outputs of the softmax statistics (any pointer but top1 may be NULL).
struct ConfOut {
  int32_t* top1 = nullptr;
  float* p1 = nullptr;    // top-1 probability
  float* p2 = nullptr;    // top-2 probability
  float* ent = nullptr;   // marginal entropy H (nats)
  float* conf = nullptr;  // the confidence the thresholds see: p1 (mode 0) or exp(-H) (mode 1)
  int mode = 0;
};
// part: [rows][nblk] {max, sum exp(z - max), id, second max}; upart: [rows][nblk] entropy
// partials (sum of e * y, y = (z - max) log2 e) or NULL (then H is not available).
cudaError_t lmhead_combine_launch(const float4* part, const float* upart, int rows, int nblk, const ConfOut& o,
                                  const int* rows_dev, const int* slot, cudaStream_t stream);
struct DcvParams {
  float tau_commit, tau_draft;
  int window, min_commit, contiguous_drafts;
  int acceptance = 0;  // 0: DCV (Eq. compute_k + Eq. draft_update); 1: Eq. threshold_pd
  int block_len = 0;   // acceptance 1: the semi-autoregressive block the rule applies to
};
// One step's acceptance on the generation rows: ids/c (and ent) are [batch][M] (position
// N + i).  With ent, jpde[b] accumulates Eq. entropy_bound of the set row b commits.
// cmt: committed flags [batch][N + M] (read and written with acceptance 1 only).
// kcap (may be NULL): per-row cap on K (RowPlan::kcap).
cudaError_t dcv_commit_launch(int32_t* x, int32_t* p, int32_t* k_out, int32_t* steps,
                              const int32_t* ids, const float* c, const float* ent, float* jpde, int batch,
                              int N, int M, const DcvParams& prm, int32_t* done_count, uint8_t* cmt,
                              const int* kcap, cudaStream_t stream);
// Block acceptance from bf16 logits (dcl_accept): c1 = p1 (mode 0) or exp(-H) (mode 1).
cudaError_t accept_stats_launch(const __nv_bfloat16* logits, const int32_t* committed, int B,
                                int P, int V, int32_t* ids, float* c1, float* c2, int mode,
                                cudaStream_t stream);
cudaError_t accept_commit_launch(const int32_t* committed, const int32_t* ids, const float* c1,
                                 int32_t* x, int32_t* k, int B, int P, const DcvParams& prm,
                                 cudaStream_t stream);
// One launch of a kernel that does only the dependent-launch handshake (launch floor).
cudaError_t empty_launch(cudaStream_t stream);
// Counter-based weight generator (SplitMix64 + Irwin-Hall(4)), with an optional
// row remap: element e of a [rows][cols] tensor goes to
// dst[(e/cols) / blk * blk_stride + blk_off + (e/cols) % blk) * cols + e % cols]
// (blk = 0 means contiguous).
cudaError_t generate_launch(__nv_bfloat16* dst, uint64_t seed, int tid, int64_t start,
                            int64_t count, float std, float mean, int64_t cols, int blk,
                            int blk_stride, int blk_off, cudaStream_t stream);
// cos / sin of the rotate-half angles t * theta^(-2j/hd), computed in double on the host,
// laid out [hd/2][T] (positions contiguous).
cudaError_t rope_table_build(float* cos_dev, float* sin_dev, int T, int hd, float theta,
                             cudaStream_t stream);

// Message returned by dcl_last_error(NULL) for calls that have no context.
void set_thread_error(const char* msg);

}  // namespace dcl
