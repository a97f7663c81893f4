/*
 * dcleap.h - C ABI of libdcleap.so: the DC-Leap denoise step of a masked-diffusion
 * LM on one NVIDIA GB300 (sm_103a), in hand-written CUDA.
 *
 * The calls follow the paper's statement of the problem: Algorithm 1 takes a model,
 * a prompt, a generation length, a maximum window size L and the two thresholds
 * (tau_commit, tau_draft) and returns the sequence x.  One denoise step is the
 * four-step iteration of Sec. 3.3: (i) re-mask the window [p, p+L) (Eq. remasking),
 * (ii) one bidirectional forward giving per-position softmax confidences (Eq. 2),
 * (iii) K by the prefix-product rule (Eq. compute_k), (iv) commit x[p:p+K] and
 * refresh drafts at every position >= p+L (Eq. draft_update); then p += K.
 *
 * Conventions (all calls):
 *   - Every call returns a dcl_status and never aborts the process; on failure the
 *     message is available from dcl_last_error(ctx).
 *   - Pointers named *_dev are device pointers owned by the caller; pointers without
 *     that suffix are host pointers owned by the caller.  The library does not check
 *     where a *_dev pointer lives or how long its buffer is (sizes follow from the
 *     call's arguments): a host pointer or a short buffer there is a device-side memory
 *     fault, not a status.  The Python binding refuses both before calling in.  The
 *     context owns every device buffer it allocates (weights, activations, scratch)
 *     and frees them in dcl_destroy.
 *   - Work is stream-ordered on the stream given to dcl_create.  Calls that return
 *     host data (dcl_step with k_out, dcl_generate, dcl_get_state) synchronise that
 *     stream; the others are asynchronous.
 *   - Token ids are int32 in [0, vocab).  Matrices are row-major bf16 in the
 *     nn.Linear layout [out_features][in_features].
 *   - Decisions compare float32 confidences with float32 thresholds, strictly (>).
 */
#ifndef DCLEAP_H
#define DCLEAP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DCL_OK = 0,
  DCL_ERR_INVALID_ARG = 1, /* a NULL/negative/oversized argument or an out-of-range id */
  DCL_ERR_STATE = 2,       /* call out of order (e.g. dcl_step before dcl_set_prompt) */
  DCL_ERR_OOM = 3,         /* device allocation failed */
  DCL_ERR_CUDA = 4,        /* a CUDA runtime/driver error, or a kernel-reported fault */
  DCL_ERR_TIMEOUT = 5,     /* dcl_generate ran max_steps without finishing, or a device-side
                              bounded wait gave up (the kernel returned without hanging) */
  DCL_ERR_UNSUPPORTED = 6  /* a shape the kernels do not support (see dcl_create) */
} dcl_status;

/* Transformer shape (Sec. 2.1: one bidirectional network over prompt + generation).
 * Supported: head_dim in {64, 128}; d_model, ffn_dim multiples of 128;
 * n_heads a multiple of n_kv_heads; (n_heads + n_kv_heads) * head_dim a multiple of 128. */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab, mask_id;
  float rope_theta, rms_eps;
} dcl_model_config;

/* Decoding hyper-parameters (Algorithm 1 inputs; defaults of Sec. 4.1 in comments). */
typedef struct {
  float tau_commit;          /* 0.70: commit threshold of Eq. compute_k (strict >) */
  float tau_draft;           /* 0.98: draft threshold of Eq. draft_update (strict >) */
  int32_t max_window;        /* L; 0 means gen_len / 2 */
  int32_t block_len;         /* 32: semi-autoregressive block length */
  int32_t gen_len;           /* M, the number of generated positions */
  int32_t kv_cache;          /* 0: full recompute every step; 1: approximate prefix key /
                                value cache refreshed at block boundaries: between refreshes a
                                step computes the positions from the block-aligned prefix end
                                N + block_len * floor((p - N) / block_len) to the end, against
                                the stored keys / values of the rest; 2: dual (prefix + suffix)
                                cache, a serving refinement outside the paper: refreshes as 1,
                                between refreshes only the current block (block_len positions
                                from the prefix end) is computed, the other generation positions
                                keep the predictions of the last refresh, and K is capped at
                                the block end (commits use fresh predictions only); acceptance
                                0 only */
  int32_t min_commit;        /* 1: K = max(K, min_commit) so every step makes progress;
                                0 keeps the literal rule (may stall; bounded by max_steps) */
  int32_t contiguous_drafts; /* 0; 1 = App. E variant (drafts only as an unbroken chain) */
  int32_t confidence;        /* 0: c = top-1 probability (Eq. threshold_pd, the paper's choice);
                                1: c = exp(-H), H = -sum_v P(v) ln P(v) the marginal entropy of
                                Eq. entropy_bound (an alternative confidence, cf. App. F.3);
                                exp(-H) <= p1, so it never accepts more than 0 */
  int32_t acceptance;        /* 0: DCV, the contiguous rule (Eq. compute_k + Eq. draft_update);
                                1: the non-contiguous rule DC-Leap is contrasted with
                                (Eq. threshold_pd, Sec. 2.1): every masked position of the
                                current semi-autoregressive block (block_len positions from
                                N + block_len * floor((p - N) / block_len), p the leftmost
                                uncommitted position) with c > tau_commit is committed at once;
                                if fewer than min_commit pass, the min_commit most confident
                                masked positions of the block are (ties to the lower position;
                                tau_commit >= 1 gives the base sampler's low-confidence
                                remasking, min_commit tokens per step); no drafts, no
                                re-masking, tau_draft / max_window / contiguous_drafts unused,
                                and K is the number committed */
} dcl_decode_config;

typedef struct {
  int64_t steps;      /* denoise iterations run */
  int64_t tokens;     /* generated tokens committed (all rows) */
  double elapsed_ms;  /* wall time of dcl_generate, host clock */
  int32_t done;       /* 1 if every row reached p = N + M */
  double jpde_bound;  /* Eq. entropy_bound (sum_U H - max_U H, nats) of every set U = [p, p+K)
                         committed in parallel since dcl_set_prompt / dcl_restart /
                         dcl_set_state, summed over steps and rows (fp32 per row) */
} dcl_stats;

/* Optional device allocator (e.g. a framework's caching allocator). */
typedef struct {
  void* (*alloc)(size_t bytes, void* user); /* returns a device pointer or NULL */
  void (*free)(void* ptr, void* user);
  void* user;
} dcl_allocator;

/* Weight kinds for dcl_set_weight (shapes with H = n_heads, G = n_kv_heads, hd =
 * head_dim, d = d_model, F = ffn_dim, V = vocab). */
typedef enum {
  DCL_W_EMBED = 0,      /* [V][d]     token embedding           (global) */
  DCL_W_ATTN_NORM = 1,  /* [d]        RMSNorm gain before attention */
  DCL_W_Q = 2,          /* [H*hd][d] */
  DCL_W_K = 3,          /* [G*hd][d] */
  DCL_W_V = 4,          /* [G*hd][d] */
  DCL_W_O = 5,          /* [d][H*hd] */
  DCL_W_MLP_NORM = 6,   /* [d]        RMSNorm gain before the MLP */
  DCL_W_GATE = 7,       /* [F][d]     SwiGLU gate */
  DCL_W_UP = 8,         /* [F][d]     SwiGLU up */
  DCL_W_DOWN = 9,       /* [d][F] */
  DCL_W_FINAL_NORM = 10,/* [d]        final RMSNorm gain        (global) */
  DCL_W_LM_HEAD = 11    /* [V][d]     untied LM head            (global) */
} dcl_weight_kind;

typedef struct dcl_ctx dcl_ctx;

/* Create a context on the current CUDA device.
 *   cfg        model shape, or NULL for an ops-only context (dcl_accept, dcl_op_*).
 *   max_batch  largest batch (rows) later passed to dcl_set_prompt.
 *   max_seq    largest N + M later passed to dcl_set_prompt.
 *   cuda_stream a cudaStream_t that all work goes to; NULL makes the context create and
 *              own a blocking stream (ordered with the legacy default stream).  The
 *              step is captured into a CUDA graph on this stream, so it must not be the
 *              legacy default stream itself.
 *   alloc      optional allocator; NULL uses cudaMalloc/cudaFree.
 * Weights are allocated (uninitialised) here: 2 bytes per parameter.
 * Errors: INVALID_ARG, UNSUPPORTED (shape), OOM, CUDA.  *out is NULL on failure. */
dcl_status dcl_create(const dcl_model_config* cfg, int32_t max_batch, int32_t max_seq,
                      void* cuda_stream, const dcl_allocator* alloc, dcl_ctx** out);

/* Copy one weight tensor (bf16, layout above) into the context; `layer` is ignored for
 * global tensors.  src is a host pointer (src_is_device = 0) or a device pointer (1).
 * The context keeps its own copy (re-laid out internally).  Errors: INVALID_ARG, CUDA. */
dcl_status dcl_set_weight(dcl_ctx* ctx, int32_t kind, int32_t layer, const void* src,
                          int32_t src_is_device);

/* Fill every weight on the device from the counter-based generator of the synthetic
 * workloads (SplitMix64 of seed<<48 | tensor<<32 | index, sum of four 16-bit fields,
 * scaled to `std`, rounded to bf16).  The LM head uses std * lm_head_scale; RMSNorm
 * gains are 1 + the same draw scaled to norm_gain_std.  seed < 65536.  Async. */
dcl_status dcl_init_random_weights(dcl_ctx* ctx, uint64_t seed, float std, float lm_head_scale,
                                   float norm_gain_std);

/* Algorithm 1 initialisation: x = prompt ++ [MASK]^M and p = N for every row
 * (Eq. 1).  prompt is host int32 [batch][n_prompt]; batch <= max_batch,
 * n_prompt + cfg->gen_len <= max_seq.  Validates ids, uploads the state and builds
 * (or reuses) the CUDA graph of one step for this shape.
 * Errors: INVALID_ARG (also kv_cache outside {0, 1, 2}, confidence or acceptance outside
 * {0, 1}, or acceptance = 1 with block_len < 1), UNSUPPORTED (kv_cache = 1 or 2 with N, M or
 * block_len not a multiple of 32; kv_cache = 2 with acceptance = 1), CUDA. */
dcl_status dcl_set_prompt(dcl_ctx* ctx, int32_t batch, const int32_t* prompt, int32_t n_prompt,
                          const dcl_decode_config* cfg);

/* One denoise step (Sec. 3.3 steps (i)-(iv) and the advance), one CUDA-graph launch on
 * the context stream.  Rows already finished are left unchanged.  If k_out is not
 * NULL it receives the K of every row (host int32 [batch]; the call synchronises).
 * Errors: STATE (no prompt), CUDA. */
dcl_status dcl_step(dcl_ctx* ctx, int32_t* k_out);

/* Run steps until every row has p = N + M (Algorithm 1's loop) or max_steps steps
 * have run.  out (host int32 [batch][M], may be NULL) receives x[N:N+M]; st (may be
 * NULL) the counters.  Synchronises.  Errors: STATE, CUDA, TIMEOUT (max_steps reached;
 * out still holds the partial result). */
dcl_status dcl_generate(dcl_ctx* ctx, int32_t max_steps, int32_t* out, dcl_stats* st);

/* Reset the decoding state to the one the last dcl_set_prompt made (x = prompt ++ MASK,
 * p = N, counters 0), asynchronously on the context stream (device-to-device copies; no
 * host synchronisation).  Lets a caller run generations of the same prompt back to back.
 * Errors: STATE, CUDA. */
dcl_status dcl_restart(dcl_ctx* ctx);

/* Read / write the decoding state (x: host int32 [batch][N+M], p: host int32 [batch]),
 * e.g. to resume a run or to drive teacher-forced parity.  get synchronises.
 * set validates ids and N <= p <= N+M; under acceptance = 1 a position counts as committed
 * when it lies before p or holds a token other than MASK.  Errors: STATE, INVALID_ARG, CUDA. */
dcl_status dcl_get_state(dcl_ctx* ctx, int32_t* x, int32_t* p);
dcl_status dcl_set_state(dcl_ctx* ctx, const int32_t* x, const int32_t* p);

/* Parity hook: step (i) and (ii) only (re-mask, forward, confidence) on the current
 * state, without committing.  Any output may be NULL:
 *   logits_dev bf16 [batch][M][V] logits of the generation rows (an extra plain GEMM),
 *   top1_dev int32 [batch][M], p1_dev / p2_dev float [batch][M] (top-1 / top-2
 *   probabilities), conf_dev float [batch][M] (the confidence the thresholds see: p1, or
 *   exp(-H) with confidence = 1), entropy_dev float [batch][M] (marginal entropy H in
 *   nats), all from the fused LM-head epilogue (the values the step itself uses).
 * Errors: STATE, CUDA. */
dcl_status dcl_forward_debug(dcl_ctx* ctx, void* logits_dev, int32_t* top1_dev, float* p1_dev,
                             float* p2_dev, float* conf_dev, float* entropy_dev);

/* Parity hook: the residual stream after the embedding (layer = -1) or after
 * transformer block `layer` of the last forward, copied to h_dev (float [batch*(N+M)][d]).
 * Call after dcl_forward_debug or dcl_forward_debug_from.  Errors: STATE, INVALID_ARG, CUDA. */
dcl_status dcl_debug_hidden(dcl_ctx* ctx, int32_t layer, float* h_dev);

/* Parity hook for per-block teacher forcing (Eq. 2's forward, one block at a time): the
 * forward of step (ii) started at transformer block `layer` (0 <= layer <= n_layers) from
 * the caller's residual stream h_dev (float [batch*(N+M)][d], row b*(N+M) + t: the stream
 * entering that block; layer = n_layers runs only the final RMSNorm and the LM head), on
 * the current state's rows, without re-mask or embedding.  Outputs as dcl_forward_debug
 * (any may be NULL); dcl_debug_hidden then reads the stream after each later block.  With
 * commit = 1 the step's acceptance (steps (iii)-(iv) and the advance of p) then runs on
 * these predictions, as in dcl_step.  Full recompute only, every sequence unfinished.
 * Synchronises.  Errors: STATE (no prompt, or a finished sequence), INVALID_ARG,
 * UNSUPPORTED (kv_cache != 0), CUDA. */
dcl_status dcl_forward_debug_from(dcl_ctx* ctx, int32_t layer, const float* h_dev, int32_t commit,
                                  void* logits_dev, int32_t* top1_dev, float* p1_dev, float* p2_dev,
                                  float* conf_dev, float* entropy_dev);

/* Acceptance pass of one block from given logits (Eq. 2 confidence + Eq. compute_k +
 * Eq. draft_update), for B independent rows of P positions:
 *   logits_dev    bf16 [B][P][V]; only uncommitted positions are read.
 *   committed_dev int32 [B]: c_b positions already committed (left-aligned), so the
 *                 window starts at p = c_b; rows with c_b >= P are left unchanged.
 *   x_dev         int32 [B][P], in/out: receives the committed ids and new drafts.
 *   cfg           thresholds, max_window (0 = P/2), min_commit, contiguous_drafts,
 *                 confidence (0: top-1 probability, 1: exp(-H) of the marginal entropy),
 *                 acceptance (0: DCV; 1: Eq. threshold_pd over the uncommitted positions
 *                 [c_b, P), K = the number committed, no drafts).
 *   k_dev         int32 [B] out: K of every row.
 * Committed c_b and repeated calls: K depends on the logits and c_b only, so a second
 * call on its own output writes the same x.  Async on the context stream; 1 <= B,
 * 1 <= P <= 4096, B*P <= 1<<20, V >= 2.  Errors: INVALID_ARG (NULL pointer, sizes,
 * confidence not 0/1), OOM (scratch), CUDA. */
dcl_status dcl_accept(dcl_ctx* ctx, const void* logits_dev, int32_t B, int32_t P, int32_t V,
                      const int32_t* committed_dev, int32_t* x_dev, const dcl_decode_config* cfg,
                      int32_t* k_dev);

/* ---- allocation-free acceptance ---- */

/* Largest B*P that dcl_accept_noalloc accepts: the size of its static scratch. */
#define DCL_NOALLOC_MAX_POSITIONS 32768

/* The paper has no counterpart of this call; it exists for callers that cannot allocate
 * device memory - code running inside another framework's memory pool, or under a
 * real-time budget where cudaMalloc may stall or is forbidden - and so cannot create a
 * dcl_ctx either.  It computes exactly what dcl_accept computes (same arguments, same
 * kernels) on `cuda_stream` (NULL = the legacy default stream), without a context and
 * without any allocation: its scratch (12 bytes per position) is a file-scope device
 * array of DCL_NOALLOC_MAX_POSITIONS positions (384 KB) that every GPU loading this
 * library holds until the process exits.
 *   - The size limits are dcl_accept's (1 <= P <= 4096, V >= 2), and B*P at most
 *     DCL_NOALLOC_MAX_POSITIONS; anything else is rejected with DCL_ERR_INVALID_ARG.
 *   - The first call on a device looks up the array's device address (once per device,
 *     with that device current) and keeps it for the life of the process; make that
 *     first call before any stream capture.  A cudaDeviceReset unloads the library's
 *     device code, array included, and leaves the kept address stale: do not call this
 *     function after one.
 *   - All calls share the one array and it keeps the last call's contents; a call
 *     writes every scratch entry it reads, so nothing needs clearing, but calls whose
 *     work overlaps on the GPU (e.g. on two streams) race on it.
 *   - Errors: INVALID_ARG, CUDA; the message is available from dcl_last_error(NULL). */
dcl_status dcl_accept_noalloc(const void* logits_dev, int32_t B, int32_t P, int32_t V,
                              const int32_t* committed_dev, int32_t* x_dev,
                              const dcl_decode_config* cfg, int32_t* k_dev, void* cuda_stream);

/* ---- FP8 weight storage (host only) ---- */

/* FP8 weights for the weight-streaming steps: a serving refinement outside the paper.
 * Quantises a bf16 weight w [rows][cols] in the nn.Linear layout (host, bf16 bit
 * patterns) to codes [rows][cols] (host, uint8) and exps [rows] (host, int32) so that row
 * n stores w[n][k] ~ value(codes[n][k]) * 2^exps[n]:
 *   - codes are E4M3 as in the OCP 8-bit floating-point specification (sign bit, four
 *     exponent bits with bias 7, three mantissa bits, exponent field 0 the subnormals
 *     m * 2^-9, no infinities, 448 the largest magnitude), each the nearest value to
 *     w[n][k] / 2^exps[n] with ties to the even mantissa and the sign kept;
 *   - exps[n] is the least integer with max_k |w[n][k]| <= 448 * 2^exps[n] (0 for a row
 *     of zeros), so every scaled row fits and its maximum lands in [224, 448];
 *   - value(code) * 2^exps[n] is then exactly representable in bf16 whenever
 *     exps[n] >= -124 (every row whose largest magnitude exceeds 2^-116).
 * Runs on the calling thread, no context and no GPU.  Errors: DCL_ERR_INVALID_ARG for a
 * NULL pointer, rows or cols < 1, or a NaN / infinite weight (message from
 * dcl_last_error(NULL)). */
dcl_status dcl_fp8_quantise(const uint16_t* w, int64_t rows, int64_t cols, uint8_t* codes, int32_t* exps);

/* ---- single-kernel entry points (the kernels of the step, for parity tests) ---- */

/* y = x / sqrt(mean(x^2) + eps) * gain.  x_dev float [rows][d], gain_dev bf16 [d],
 * y_dev bf16 [rows][d]; d a multiple of 4.  Async. */
dcl_status dcl_op_rmsnorm(dcl_ctx* ctx, const float* x_dev, const void* gain_dev, void* y_dev,
                          int32_t rows, int32_t d, float eps);

/* Tile choices of the GEMM entry points: 0 lets the library choose (as in the step),
 * 128 / 256 force a one-CTA 128 x 128 / 128 x 256 tile, DCL_TILE_PAIR a CTA-pair
 * (tcgen05 cta_group::2) 256 x 256 tile with the library's choice of K splitting,
 * DCL_TILE_PAIR | (S << 8) that tile with the K dimension split S ways (S = 1: unsplit),
 * DCL_TILE_PAIR | DCL_TILE_STREAMK | (S << 8) that tile with the stream-K schedule: the
 * tiles of a partly filled last round of the persistent grid are cut into about S K
 * segments each (S = 0: shared out over all CTA pairs) run by different pairs; rejected
 * with DCL_ERR_INVALID_ARG when the last round is full or a sharing pair would get no K
 * block; DCL_TILE_PAIR | DCL_TILE_HALVES whole tiles in full rounds, then every tile of a partial
 * last round as two 256 x 128 pieces (no K split); DCL_TILE_PAIR | DCL_TILE_DSMEM clusters
 * of two CTA pairs: whole tiles in full rounds, then every left-over tile split by K over
 * one cluster's pairs, the upper half's fp32 sum added to the lower half's through
 * distributed shared memory (K >= 128, at most one left-over tile per cluster).
 * Partial sums are always combined in K order, so every choice is deterministic. */
#define DCL_TILE_PAIR 2
#define DCL_TILE_STREAMK (1 << 16)
#define DCL_TILE_HALVES (1 << 18)
#define DCL_TILE_DSMEM (1 << 19)

/* The dense contractions of the forward (Sec. 3.3 step (ii)): out = a @ w^T on the tcgen05
 * tensor cores.  a_dev bf16 [M][K], w_dev bf16 [N][K];
 * mode 0: out bf16 [M][N]; mode 1: out float [M][N] += a @ w^T (residual add).
 * K a multiple of 64, N of 32.  Synchronises (reports device-side faults). */
dcl_status dcl_op_linear(dcl_ctx* ctx, const void* a_dev, const void* w_dev, void* out_dev,
                         int32_t M, int32_t N, int32_t K, int32_t mode, int32_t tile);

/* Non-causal attention softmax(q k^T / sqrt(hd)) v over all T positions of each of
 * `batch` sequences (the attention of the bidirectional pass, Eq. 2).  qkv_dev bf16
 * [batch*T][(H+2G)*hd] (q | k | v column blocks, RoPE already applied), out_dev bf16
 * [batch*T][H*hd]; both 16-byte aligned.  hd in {64, 128}.  q_rows > 0 (a multiple of 32,
 * at most T) takes as queries only the last q_rows positions of each sequence (rows
 * b*T + T - q_rows onwards), which attend to all T positions, and writes only those
 * output rows (the suffix rows of a step with the key / value cache); 0 takes all T.
 * Synchronises. */
dcl_status dcl_op_attention(dcl_ctx* ctx, const void* qkv_dev, void* out_dev, int32_t batch,
                            int32_t T, int32_t H, int32_t G, int32_t hd, int32_t q_rows);

/* LM head + softmax confidence fused (Eq. 2; top-1 of Eq. threshold_pd; top-2 of
 * Sec. 2.2): for each row r of x_dev (bf16 [R][d]), z = x_r @ w^T (w_dev bf16 [V][d]);
 * top1_dev[r] = argmax (lowest index on ties), p1_dev[r] = max softmax(z), p2_dev[r] =
 * second largest probability, entropy_dev[r] (may be NULL) = -sum_v P(v) ln P(v) (nats,
 * the per-token entropy of Eq. entropy_bound).  Logits never reach memory.  d a multiple
 * of 64; tile 0, 256 or DCL_TILE_PAIR.  Synchronises. */
dcl_status dcl_op_lmhead_top2(dcl_ctx* ctx, const void* x_dev, const void* w_dev, int32_t R,
                              int32_t V, int32_t d, int32_t* top1_dev, float* p1_dev,
                              float* p2_dev, float* entropy_dev, int32_t tile);

/* Fill dst_dev (bf16, count elements) from the weight generator of
 * dcl_init_random_weights for tensor id `tid` starting at element `start`.  Async. */
dcl_status dcl_op_generate(dcl_ctx* ctx, void* dst_dev, uint64_t seed, int32_t tid, int64_t start,
                           int64_t count, float std, float mean);

/* ---- per-kernel timing of the step graph ---- */

/* Kernel classes reported by dcl_profile_last_step. */
typedef enum {
  DCL_K_EMBED = 0,       /* remask + embedding gather */
  DCL_K_RMSNORM = 1,
  DCL_K_GEMM_QKV = 2,    /* QKV projection + RoPE epilogue */
  DCL_K_ATTENTION = 3,
  DCL_K_GEMM_O = 4,      /* output projection + residual */
  DCL_K_GEMM_GATEUP = 5, /* gate/up projection + SwiGLU */
  DCL_K_GEMM_DOWN = 6,   /* down projection + residual */
  DCL_K_GEMM_LMHEAD = 7, /* LM head + softmax/top-2 partials */
  DCL_K_COMBINE = 8,     /* merge of the LM-head partials */
  DCL_K_DCV = 9,         /* commit / draft / advance */
  DCL_K_VTRANSPOSE = 10, /* v written transposed for the attention kernel */
  DCL_K_ROWPLAN = 11,    /* the rows the step computes (full recompute or cache suffix) */
  DCL_K_GEMM_MLP = 12    /* gate/up + SwiGLU and down + residual as one launch (the step's
                            default; the two launches above when the fusion is off) */
} dcl_kernel_kind;

/* Fault-handling self-test (the device waits of the GEMM and attention pipelines are
 * bounded; this exercises that path without a fault): a one-thread kernel waits on
 * something nothing signals - which = 0: a fresh mbarrier, 1: a zero counter in global
 * memory - through the same bounded helpers, gives up after the 2 s wait limit and
 * records the timeout.  Returns DCL_ERR_TIMEOUT (the expected outcome) and leaves the
 * context usable; INVALID_ARG for another `which`.  Synchronises. */
dcl_status dcl_selftest_wait_timeout(dcl_ctx* ctx, int32_t which);

/* Launch floor of a step: a CUDA graph of n_kernels launches of an empty kernel (each
 * one does only the dependent-launch handshake the step's kernels do, launched with the
 * same programmatic-serialisation attribute) is captured on the context stream, launched
 * 3 times untimed and `reps` times between CUDA events; *ms_per_graph receives the mean
 * time of one graph.  A step of n_kernels launches cannot run faster.  Synchronises.
 * Errors: INVALID_ARG (n_kernels outside [1, 100000], reps < 1, NULL output), CUDA. */
dcl_status dcl_launch_floor(dcl_ctx* ctx, int32_t n_kernels, int32_t reps, float* ms_per_graph);

/* enable = 1 re-captures the step graph with a pair of timing events (CUDA event record
 * nodes on the context stream) around every kernel; 0 restores the plain graph.
 * Takes effect at once if a prompt is set, else at the next dcl_set_prompt. */
dcl_status dcl_set_profiling(dcl_ctx* ctx, int32_t enable);

/* Per-kernel device durations (ms) of the most recent step run with profiling on, in
 * launch order: ms[i], kind[i] for i < *n (at most cap).  Synchronises.
 * Errors: STATE (profiling off or no step yet), CUDA. */
dcl_status dcl_profile_last_step(dcl_ctx* ctx, float* ms, int32_t* kind, int32_t cap, int32_t* n);

/* Last error message of this context (or of the last failed dcl_create when ctx is NULL). */
const char* dcl_last_error(const dcl_ctx* ctx);

/* Free everything the context owns.  NULL is a no-op. */
void dcl_destroy(dcl_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* DCLEAP_H */
