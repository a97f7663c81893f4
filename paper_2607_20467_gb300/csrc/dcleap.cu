// C ABI of libdcleap.so (include/dcleap.h): the context, weight layout, the captured
// CUDA graph of one denoise step (Sec. 3.3 steps (i)-(iv), Algorithm 1), the host
// loop of Algorithm 1, and single-kernel entry points for parity tests.
#include <algorithm>
#include <chrono>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/dcleap.h"
#include "common.cuh"

using namespace dcl;

namespace {

thread_local std::string g_create_error;

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

struct Layer {
  __nv_bfloat16 *attn_norm, *wqkv, *wo, *mlp_norm, *wgu, *wdown;
};

struct Launch {  // one kernel launch of the step, for profiling
  int kind;
  cudaEvent_t start, stop;
};

}  // namespace

struct dcl_ctx {
  bool has_model = false;
  dcl_model_config cfg{};
  int max_batch = 0, max_seq = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  dcl_allocator alloc{};
  bool custom_alloc = false;
  int num_sms = 0;
  std::string err;
  std::vector<void*> owned;

  // weights (one allocation)
  void* wbuf = nullptr;
  __nv_bfloat16 *embed = nullptr, *final_norm = nullptr, *lm_head = nullptr;
  std::vector<Layer> layers;

  // activations, sized for max_batch * max_seq rows
  float* h = nullptr;
  __nv_bfloat16 *xn = nullptr, *qkv = nullptr, *attn = nullptr, *act = nullptr, *xg = nullptr;
  __half* vt = nullptr;           // v transposed (fp16) for the attention kernel (full recompute)
  __nv_bfloat16* kbuf = nullptr;  // keys after RoPE [B][T][G*hd] (full recompute)
  __nv_bfloat16* kvstore = nullptr;  // approximate cache: per layer keys [B][T][G*hd], v^T
  size_t kvstore_bytes = 0;
  int* rp_buf = nullptr;          // the row plan's tables
  RowPlan rp;
  float4* part = nullptr;
  float* ent_part = nullptr;  // LM-head entropy partials [rows][tiles]
  int32_t* top1 = nullptr;
  float *p1 = nullptr, *p2 = nullptr;
  float* ent = nullptr;   // marginal entropy H of every generation position
  float* conf = nullptr;  // exp(-H) (the thresholds' input with confidence = 1)
  float* jpde = nullptr;  // per row: Eq. entropy_bound summed over the committed sets
  int32_t *x = nullptr, *p = nullptr, *k = nullptr, *steps = nullptr, *done_count = nullptr;
  int32_t *x_init = nullptr, *p_init = nullptr;  // state at the last dcl_set_prompt
  uint8_t *cmt = nullptr, *cmt_init = nullptr;    // committed flags [B][T] (Eq. threshold_pd decoding)
  int* derr = nullptr;
  float *rope_cos = nullptr, *rope_sin = nullptr;
  float* snap = nullptr;  // residual stream after the embedding and after each layer (debug)
  int* gemm_flags = nullptr;  // split-K counters of the step's GEMMs (zero between launches)
  size_t gemm_flags_n = 0;
  float* gemm_ws = nullptr;   // split-K partials of the step's GEMMs
  size_t gemm_ws_n = 0;
  size_t snap_rows = 0;

  // accept scratch (dcl_accept)
  int32_t* acc_ids = nullptr;
  float *acc_c1 = nullptr, *acc_c2 = nullptr;
  size_t acc_cap = 0;

  // per-shape state
  bool prompt_set = false;
  int B = 0, N = 0, M = 0, T = 0, window = 0;
  dcl_decode_config dcfg{};
  std::vector<GemmPlan> plans;  // 4 per layer + LM head
  std::vector<AttnPlan> attn_plans;  // one per layer
  bool kv_fused = false;  // the QKV GEMMs write k and v^T (no transpose launch)
  cudaGraphExec_t gexec = nullptr;
  bool profiling = false;
  std::vector<Launch> launches;
  size_t launch_i = 0;
  bool profiled_step = false;
  int32_t* h_done = nullptr;  // pinned [2]
  cudaEvent_t ev_done[2] = {nullptr, nullptr};
};

namespace {

dcl_status fail(dcl_ctx* c, dcl_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (c)
    c->err = buf;
  else
    g_create_error = buf;
  return s;
}

#define CUDA_TRY(ctx, expr)                                                                  \
  do {                                                                                       \
    cudaError_t e_ = (expr);                                                                 \
    if (e_ != cudaSuccess)                                                                   \
      return fail((ctx), DCL_ERR_CUDA, "%s failed: %s", #expr, cudaGetErrorString(e_));     \
  } while (0)

void* dev_alloc(dcl_ctx* c, size_t bytes) {
  void* ptr = nullptr;
  if (bytes == 0) bytes = 16;
  if (c->custom_alloc) {
    ptr = c->alloc.alloc(bytes, c->alloc.user);
  } else if (cudaMalloc(&ptr, bytes) != cudaSuccess) {
    cudaGetLastError();
    ptr = nullptr;
  }
  if (ptr) c->owned.push_back(ptr);
  return ptr;
}

void release_stream(dcl_ctx* c) {
  if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
  c->stream = nullptr;
  c->own_stream = false;
}

void dev_free_all(dcl_ctx* c) {
  for (void* ptr : c->owned) {
    if (c->custom_alloc)
      c->alloc.free(ptr, c->alloc.user);
    else
      cudaFree(ptr);
  }
  c->owned.clear();
}

void dev_free_one(dcl_ctx* c, void* ptr) {
  if (!ptr) return;
  for (size_t i = 0; i < c->owned.size(); ++i) {
    if (c->owned[i] == ptr) {
      c->owned.erase(c->owned.begin() + i);
      if (c->custom_alloc)
        c->alloc.free(ptr, c->alloc.user);
      else
        cudaFree(ptr);
      return;
    }
  }
}

// Read and clear the device error word; map it to a status.
dcl_status check_device(dcl_ctx* c) {
  int e = 0;
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  CUDA_TRY(c, cudaMemcpy(&e, c->derr, sizeof(int), cudaMemcpyDeviceToHost));
  if (e != DERR_NONE) {
    const int zero = 0;
    cudaMemcpy(c->derr, &zero, sizeof(int), cudaMemcpyHostToDevice);
    // an aborted split-K launch may leave its counters set: clear them for the next one
    if (c->gemm_flags) cudaMemset(c->gemm_flags, 0, sizeof(int) * c->gemm_flags_n);
    if (e == DERR_WAIT_TIMEOUT)
      return fail(c, DCL_ERR_TIMEOUT, "a pipeline wait timed out on the device (kernel returned)");
    if (e == DERR_TOKEN_RANGE) return fail(c, DCL_ERR_INVALID_ARG, "a token id outside [0, vocab) reached the embedding");
    return fail(c, DCL_ERR_CUDA, "device error code %d", e);
  }
  return DCL_OK;
}

// ------------------------------------------------------------------ the step
struct Enq {
  dcl_ctx* c;
  bool prof;
  cudaError_t err = cudaSuccess;
  const char* what = nullptr;
  void begin(int kind) {
    if (!prof || err != cudaSuccess) return;
    if (c->launch_i >= c->launches.size()) {
      Launch l{kind, nullptr, nullptr};
      cudaEventCreate(&l.start);
      cudaEventCreate(&l.stop);
      c->launches.push_back(l);
    }
    Launch& l = c->launches[c->launch_i];
    l.kind = kind;
    err = cudaEventRecordWithFlags(l.start, c->stream, cudaEventRecordExternal);
  }
  void end(cudaError_t e, const char* name) {
    if (err == cudaSuccess && e != cudaSuccess) {
      err = e;
      what = name;
    }
    if (!prof || err != cudaSuccess) return;
    err = cudaEventRecordWithFlags(c->launches[c->launch_i].stop, c->stream, cudaEventRecordExternal);
    ++c->launch_i;
  }
};

// Enqueue the forward (and, if with_dcv, the acceptance) on the context stream.  With
// h_in the forward starts at block first_layer from that residual stream (row b*T + t;
// no re-mask, no embedding; full recompute only).
cudaError_t enqueue_step(dcl_ctx* c, bool with_dcv, bool prof, bool snapshots, const char** what,
                         int first_layer = 0, const float* h_in = nullptr) {
  const dcl_model_config& m = c->cfg;
  const int R = c->B * c->T;
  const int d = m.d_model;
  Enq q{c, prof};
  if (prof) c->launch_i = 0;
  q.begin(DCL_K_ROWPLAN);
  q.end(row_plan_launch(c->rp, c->p, c->B, c->N, c->T, c->dcfg.block_len, c->dcfg.kv_cache, with_dcv ? 1 : 0,
                        c->x, c->dcfg.acceptance ? 0 : c->window, m.mask_id, c->stream),
        "row_plan");
  if (h_in) {
    if (q.err == cudaSuccess)
      q.err = cudaMemcpyAsync(c->h, h_in, sizeof(float) * R * d, cudaMemcpyDeviceToDevice, c->stream);
  } else {
    first_layer = 0;
    q.begin(DCL_K_EMBED);
    // (the threshold rule keeps no drafts: nothing to re-mask)
    q.end(embed_remask_launch(c->x, c->p, c->B, c->T, c->dcfg.acceptance ? 0 : c->window, m.mask_id, m.vocab,
                              c->embed, d, c->h, c->derr, c->rp, c->stream),
          "embed");
  }
  if (snapshots && q.err == cudaSuccess)
    q.err = cudaMemcpyAsync(c->snap + (size_t)first_layer * R * d, c->h, sizeof(float) * R * d,
                            cudaMemcpyDeviceToDevice, c->stream);
  for (int l = first_layer; l < m.n_layers && q.err == cudaSuccess; ++l) {
    const Layer& L = c->layers[l];
    const GemmPlan* P = &c->plans[4 * l];
    q.begin(DCL_K_RMSNORM);
    q.end(rmsnorm_launch(c->h, L.attn_norm, c->xn, R, d, m.rms_eps, c->rp.counts, nullptr, c->stream), "rmsnorm");
    q.begin(DCL_K_GEMM_QKV);
    q.end(gemm_launch(P[0], c->derr, c->stream), "gemm_qkv");
    if (!c->kv_fused) {
      q.begin(DCL_K_VTRANSPOSE);
      q.end(attention_transpose_launch(c->attn_plans[l], c->stream), "v_transpose");
    }
    q.begin(DCL_K_ATTENTION);
    q.end(attention_core_launch(c->attn_plans[l], c->derr, c->stream), "attention");
    q.begin(DCL_K_GEMM_O);
    q.end(gemm_launch(P[1], c->derr, c->stream), "gemm_o");
    q.begin(DCL_K_RMSNORM);
    q.end(rmsnorm_launch(c->h, L.mlp_norm, c->xn, R, d, m.rms_eps, c->rp.counts, nullptr, c->stream), "rmsnorm");
    if (P[2].fuse) {  // gate/up + SwiGLU and down + residual in one launch
      q.begin(DCL_K_GEMM_MLP);
      q.end(gemm_launch(P[2], c->derr, c->stream), "gemm_mlp");
    } else {
      q.begin(DCL_K_GEMM_GATEUP);
      q.end(gemm_launch(P[2], c->derr, c->stream), "gemm_gateup");
      q.begin(DCL_K_GEMM_DOWN);
      q.end(gemm_launch(P[3], c->derr, c->stream), "gemm_down");
    }
    if (snapshots && q.err == cudaSuccess)
      q.err = cudaMemcpyAsync(c->snap + (size_t)(l + 1) * R * d, c->h, sizeof(float) * R * d,
                              cudaMemcpyDeviceToDevice, c->stream);
  }
  // final norm on the computed generation rows only (LM row j <- computed row lm_src[j])
  q.begin(DCL_K_RMSNORM);
  q.end(rmsnorm_launch(c->h, c->final_norm, c->xg, c->B * c->M, d, m.rms_eps, c->rp.counts + 1, c->rp.lm_src,
                       c->stream),
        "final_rmsnorm");
  q.begin(DCL_K_GEMM_LMHEAD);
  q.end(gemm_launch(c->plans[4 * m.n_layers], c->derr, c->stream), "gemm_lmhead");
  q.begin(DCL_K_COMBINE);
  ConfOut co;
  co.top1 = c->top1;
  co.p1 = c->p1;
  co.p2 = c->p2;
  co.ent = c->ent;
  co.mode = c->dcfg.confidence;
  co.conf = co.mode ? c->conf : c->p1;
  q.end(lmhead_combine_launch(c->part, c->ent_part, c->B * c->M, gemm_lmhead_blocks(m.vocab), co, c->rp.counts + 1,
                              c->rp.lm_slot, c->stream),
        "combine");
  if (with_dcv) {
    DcvParams prm{c->dcfg.tau_commit, c->dcfg.tau_draft, c->window, c->dcfg.min_commit,
                  c->dcfg.contiguous_drafts, c->dcfg.acceptance, c->dcfg.block_len};
    q.begin(DCL_K_DCV);
    q.end(dcv_commit_launch(c->x, c->p, c->k, c->steps, c->top1, co.conf, c->ent, c->jpde, c->B, c->N, c->M, prm,
                            c->done_count, c->cmt, c->rp.kcap, c->stream),
          "dcv_commit");
  }
  if (what) *what = q.what;
  return q.err;
}

dcl_status build_graph(dcl_ctx* c) {
  if (c->gexec) {
    cudaGraphExecDestroy(c->gexec);
    c->gexec = nullptr;
  }
  cudaGraph_t g = nullptr;
  CUDA_TRY(c, cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal));
  const char* what = nullptr;
  cudaError_t e = enqueue_step(c, true, c->profiling, false, &what);
  cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
  if (e != cudaSuccess)
    return fail(c, DCL_ERR_CUDA, "capturing the step failed at %s: %s", what ? what : "?",
                cudaGetErrorString(e));
  if (e2 != cudaSuccess) return fail(c, DCL_ERR_CUDA, "end capture: %s", cudaGetErrorString(e2));
  e = cudaGraphInstantiate(&c->gexec, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(e));
  c->profiled_step = false;
  return DCL_OK;
}

// Tile of one of the step's GEMMs ("qkv", "o", "gateup", "down", "lmhead") forced by the
// environment variable DCL_GEMM_TILES, e.g. "o=128,down=pair:2" (128 / 256 = one-CTA tile
// width, pair[:S] = CTA-pair tile with S K-splits, pair:sk[:S] = CTA-pair tile with the
// stream-K schedule, S segments per left-over tile, pair:h = left-over tiles as
// half-width pieces, pair:ds =
// left-over tiles split by K over a cluster's two pairs); 0 = let the planner choose.
int tile_override(const char* name) {
  const char* env = getenv("DCL_GEMM_TILES");
  if (!env) return 0;
  const size_t n = strlen(name);
  for (const char* s = env; *s;) {
    const char* e = strchr(s, ',');
    const size_t len = e ? (size_t)(e - s) : strlen(s);
    if (len > n && strncmp(s, name, n) == 0 && s[n] == '=') {
      const char* v = s + n + 1;
      if (strncmp(v, "pair:sk", 7) == 0) return kTilePair | kTileStreamK | ((v[7] == ':' ? atoi(v + 8) : 0) << 8);
      if (strcmp(v, "pair:h") == 0 || strncmp(v, "pair:h,", 7) == 0) return kTilePair | kTileHalves;
      if (strncmp(v, "pair:ds", 7) == 0) return kTilePair | kTileDsmem;
      if (strncmp(v, "pair", 4) == 0) return kTilePair | ((v[4] == ':' ? atoi(v + 5) : 0) << 8);
      return atoi(v);
    }
    s += len + (e ? 1 : 0);
  }
  return 0;
}

dcl_status build_plans(dcl_ctx* c) {
  const dcl_model_config& m = c->cfg;
  const int R = c->B * c->T, d = m.d_model, hd = m.head_dim, H = m.n_heads, G = m.n_kv_heads;
  const int nqkv = (H + 2 * G) * hd;
  const bool cached = c->dcfg.kv_cache != 0;
  c->plans.assign(4 * m.n_layers + 1, GemmPlan{});
  const char* why = nullptr;
  // the step's GEMMs run CTA-pair tiles (their epilogues know the step's row plan); an
  // override may still ask for another tile
  auto pick = [](int t) { return t ? t : kTilePair; };
  const int t_qkv = pick(tile_override("qkv")), t_o = pick(tile_override("o")), t_gu = pick(tile_override("gateup")),
            t_down = pick(tile_override("down")), t_lm = pick(tile_override("lmhead"));
  // keys / values: one set shared by the layers (full recompute), or a set per layer kept
  // between steps (approximate cache)
  const int Tp = attn_vt_pitch(c->T);
  const size_t k_elems = (size_t)c->B * c->T * G * hd, v_elems = (size_t)c->B * G * hd * Tp;
  if (cached) {
    const size_t need = 2 * (k_elems + v_elems) * m.n_layers;
    if (need > c->kvstore_bytes) {
      CUDA_TRY(c, cudaStreamSynchronize(c->stream));
      dev_free_one(c, c->kvstore);
      c->kvstore = static_cast<__nv_bfloat16*>(dev_alloc(c, need));
      c->kvstore_bytes = c->kvstore ? need : 0;
      if (!c->kvstore) return fail(c, DCL_ERR_OOM, "key / value store allocation (%.2f GB) failed", need / 1e9);
    }
  }
  auto kbuf_of = [&](int l) { return cached ? c->kvstore + (size_t)l * (k_elems + v_elems) : c->kbuf; };
  auto vbuf_of = [&](int l) {  // (the store's v^T part holds fp16, 2 bytes per element like the keys)
    return cached ? reinterpret_cast<__half*>(c->kvstore + (size_t)l * (k_elems + v_elems) + k_elems) : c->vt;
  };
  for (int l = 0; l < m.n_layers; ++l) {
    const Layer& L = c->layers[l];
    EpiParams e0;
    e0.out = c->qkv;
    e0.ldo = nqkv;
    e0.rope_cos = c->rope_cos;
    e0.rope_sin = c->rope_sin;
    e0.rope_T = c->max_seq;
    e0.rope_cols = (H + G) * hd;
    e0.head_dim = hd;
    e0.seq_T = c->T;
    e0.m_dev = c->rp.counts;
    e0.row_pos = c->rp.row_pos;
    e0.row_seq = c->rp.row_seq;
    if (gemm_plan(&c->plans[4 * l], c->xn, R, d, L.wqkv, nqkv, EPI_QKV_ROPE, e0, c->num_sms, t_qkv, &why))
      return fail(c, DCL_ERR_UNSUPPORTED, "QKV plan: %s", why ? why : "?");
    EpiParams e1;
    e1.out = c->h;
    e1.ldo = d;
    e1.m_dev = c->rp.counts;
    if (gemm_plan(&c->plans[4 * l + 1], c->attn, R, H * hd, L.wo, d, EPI_RESID_F32, e1, c->num_sms, t_o, &why))
      return fail(c, DCL_ERR_UNSUPPORTED, "O plan: %s", why ? why : "?");
    EpiParams e2;
    e2.out = c->act;
    e2.ldo = m.ffn_dim;
    e2.m_dev = c->rp.counts;
    // the MLP as one launch (gate/up tiles, then the down projection's K-split items, each
    // waiting only for the act columns it reads), unless a tile override or DCL_MLP_FUSED=0
    // asks for the two GEMMs on their own
    const char* fenv = getenv("DCL_MLP_FUSED");
    const bool fuse_mlp = !(fenv && fenv[0] == '0') && t_gu == kTilePair && t_down == kTilePair;
    if (!fuse_mlp || gemm_plan_mlp(&c->plans[4 * l + 2], c->xn, R, d, L.wgu, m.ffn_dim, e2, L.wdown, e1,
                                   c->num_sms, &why) != cudaSuccess) {
      if (gemm_plan(&c->plans[4 * l + 2], c->xn, R, d, L.wgu, 2 * m.ffn_dim, EPI_SWIGLU, e2, c->num_sms, t_gu, &why))
        return fail(c, DCL_ERR_UNSUPPORTED, "gate/up plan: %s", why ? why : "?");
      if (gemm_plan(&c->plans[4 * l + 3], c->act, R, m.ffn_dim, L.wdown, d, EPI_RESID_F32, e1, c->num_sms, t_down,
                    &why))
        return fail(c, DCL_ERR_UNSUPPORTED, "down plan: %s", why ? why : "?");
    }
    for (int i = 0; i < 4; ++i)
      if (c->plans[4 * l + i].streamk)
        return fail(c, DCL_ERR_UNSUPPORTED, "stream-K needs a fixed row count; the step's GEMMs cannot use it");
  }
  c->kv_fused = true;
  for (int l = 0; l < m.n_layers && c->kv_fused; ++l)
    c->kv_fused = gemm_fuse_kv(&c->plans[4 * l], kbuf_of(l), vbuf_of(l), c->B, c->T, H, G, hd, Tp);
  if (!c->kv_fused) {
    if (cached) return fail(c, DCL_ERR_UNSUPPORTED, "the key / value cache needs N + M a multiple of 32");
    for (int l = 0; l < m.n_layers; ++l) {
      c->plans[4 * l].ep.vt_heads = 0;
      c->plans[4 * l].ep.k_store = 0;
    }
  }
  c->attn_plans.assign(m.n_layers, AttnPlan{});
  for (int l = 0; l < m.n_layers; ++l) {
    // (without the fused key store the rows are the identity layout b*T + t: no tables)
    if (attention_plan(&c->attn_plans[l], c->qkv, c->kv_fused ? kbuf_of(l) : nullptr, vbuf_of(l), c->attn, c->B, c->T,
                       H, G, hd, R, c->kv_fused ? c->rp.seq_off : nullptr, c->kv_fused ? c->rp.seq_len : nullptr) !=
        cudaSuccess)
      return fail(c, DCL_ERR_UNSUPPORTED, "attention plan failed");
  }
  EpiParams el;
  el.out = c->part;
  el.ent_part = c->ent_part;
  el.m_dev = c->rp.counts + 1;
  if (gemm_plan(&c->plans[4 * m.n_layers], c->xg, c->B * c->M, d, c->lm_head, m.vocab, EPI_LMHEAD, el,
                c->num_sms, t_lm, &why))
    return fail(c, DCL_ERR_UNSUPPORTED, "LM-head plan: %s", why ? why : "?");
  if (c->plans[4 * m.n_layers].streamk)
    return fail(c, DCL_ERR_UNSUPPORTED, "stream-K needs a fixed row count; the step's GEMMs cannot use it");
  // split-K counters and partials, shared by the step's GEMMs (they run one after another)
  size_t need_f = 0, need_w = 0;
  for (const GemmPlan& p : c->plans) {
    need_f = p.flags_needed > need_f ? p.flags_needed : need_f;
    need_w = p.ws_needed > need_w ? p.ws_needed : need_w;
  }
  if (need_f > c->gemm_flags_n || need_w > c->gemm_ws_n) {
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));  // no launch may still use the old buffers
    if (c->gexec) {
      cudaGraphExecDestroy(c->gexec);
      c->gexec = nullptr;
    }
  }
  if (need_f > c->gemm_flags_n) {
    dev_free_one(c, c->gemm_flags);
    c->gemm_flags = static_cast<int*>(dev_alloc(c, sizeof(int) * need_f));
    if (!c->gemm_flags) return fail(c, DCL_ERR_OOM, "split-K counter allocation failed");
    CUDA_TRY(c, cudaMemset(c->gemm_flags, 0, sizeof(int) * need_f));
    c->gemm_flags_n = need_f;
  }
  if (need_w > c->gemm_ws_n) {
    dev_free_one(c, c->gemm_ws);
    c->gemm_ws = static_cast<float*>(dev_alloc(c, sizeof(float) * need_w));
    if (!c->gemm_ws) return fail(c, DCL_ERR_OOM, "split-K workspace allocation failed");
    c->gemm_ws_n = need_w;
  }
  for (GemmPlan& p : c->plans)
    if (gemm_bind_scratch(&p, c->gemm_flags, c->gemm_ws) != cudaSuccess)
      return fail(c, DCL_ERR_CUDA, "GEMM scratch binding failed");
  return DCL_OK;
}

// Scratch for a one-off GEMM launch (the single-kernel entry points): allocated here,
// released by release_scratch after the launch has completed.
void release_scratch(dcl_ctx* c, GemmPlan* p);

dcl_status attach_scratch(dcl_ctx* c, GemmPlan* p) {
  if (p->flags_needed) {
    p->flags = static_cast<int*>(dev_alloc(c, sizeof(int) * p->flags_needed));
    if (!p->flags) return fail(c, DCL_ERR_OOM, "split-K counter allocation failed");
    CUDA_TRY(c, cudaMemsetAsync(p->flags, 0, sizeof(int) * p->flags_needed, c->stream));
  }
  if (p->ws_needed) {
    p->ws = static_cast<float*>(dev_alloc(c, sizeof(float) * p->ws_needed));
    if (!p->ws) {
      dev_free_one(c, p->flags);
      p->flags = nullptr;
      return fail(c, DCL_ERR_OOM, "split-K workspace allocation failed");
    }
  }
  if (gemm_bind_scratch(p, p->flags, p->ws) != cudaSuccess) {
    release_scratch(c, p);
    return fail(c, DCL_ERR_CUDA, "GEMM scratch binding failed");
  }
  return DCL_OK;
}

void release_scratch(dcl_ctx* c, GemmPlan* p) {
  cudaStreamSynchronize(c->stream);
  dev_free_one(c, p->flags);
  dev_free_one(c, p->ws);
  p->flags = nullptr;
  p->ws = nullptr;
}

// weight destination for (kind, layer): pointer, rows, and the gate/up interleave offset
struct WDst {
  __nv_bfloat16* ptr;
  int64_t rows, cols;
  int blk_off;  // -1: contiguous; else 0 (gate) / 128 (up) rows within each 256-row group
};

bool weight_dst(dcl_ctx* c, int kind, int layer, WDst* o) {
  const dcl_model_config& m = c->cfg;
  const int64_t d = m.d_model, hd = m.head_dim, H = m.n_heads, G = m.n_kv_heads, F = m.ffn_dim, V = m.vocab;
  const bool global = kind == DCL_W_EMBED || kind == DCL_W_FINAL_NORM || kind == DCL_W_LM_HEAD;
  if (kind < 0 || kind > DCL_W_LM_HEAD) return false;
  if (!global && (layer < 0 || layer >= m.n_layers)) return false;
  const Layer* L = global ? nullptr : &c->layers[layer];
  o->blk_off = -1;
  switch (kind) {
    case DCL_W_EMBED: *o = {c->embed, V, d, -1}; break;
    case DCL_W_ATTN_NORM: *o = {L->attn_norm, 1, d, -1}; break;
    case DCL_W_Q: *o = {L->wqkv, H * hd, d, -1}; break;
    case DCL_W_K: *o = {L->wqkv + H * hd * d, G * hd, d, -1}; break;
    case DCL_W_V: *o = {L->wqkv + (H + G) * hd * d, G * hd, d, -1}; break;
    case DCL_W_O: *o = {L->wo, d, H * hd, -1}; break;
    case DCL_W_MLP_NORM: *o = {L->mlp_norm, 1, d, -1}; break;
    case DCL_W_GATE: *o = {L->wgu, F, d, 0}; break;
    case DCL_W_UP: *o = {L->wgu, F, d, 128}; break;
    case DCL_W_DOWN: *o = {L->wdown, d, F, -1}; break;
    case DCL_W_FINAL_NORM: *o = {c->final_norm, 1, d, -1}; break;
    case DCL_W_LM_HEAD: *o = {c->lm_head, V, d, -1}; break;
  }
  return true;
}

int tensor_id(int kind, int layer) {
  const bool global = kind == DCL_W_EMBED || kind == DCL_W_FINAL_NORM || kind == DCL_W_LM_HEAD;
  return 16 * (global ? 4095 : layer) + kind;
}

dcl_status validate_ids(dcl_ctx* c, const int32_t* ids, size_t n) {
  for (size_t i = 0; i < n; ++i)
    if (ids[i] < 0 || ids[i] >= c->cfg.vocab)
      return fail(c, DCL_ERR_INVALID_ARG, "token id %d at index %zu outside [0, %d)", ids[i], i, c->cfg.vocab);
  return DCL_OK;
}

dcl_status reset_done_count(dcl_ctx* c, const int32_t* p_host) {
  int32_t n = 0;
  for (int b = 0; b < c->B; ++b) n += p_host[b] >= c->T;
  CUDA_TRY(c, cudaMemcpyAsync(c->done_count, &n, sizeof n, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  return DCL_OK;
}

}  // namespace

void dcl::set_thread_error(const char* msg) { g_create_error = msg ? msg : ""; }

// ==================================================================== C ABI
extern "C" {

const char* dcl_last_error(const dcl_ctx* ctx) {
  return ctx ? ctx->err.c_str() : g_create_error.c_str();
}

dcl_status dcl_create(const dcl_model_config* cfg, int32_t max_batch, int32_t max_seq, void* cuda_stream,
                      const dcl_allocator* alloc, dcl_ctx** out) {
  if (!out) return fail(nullptr, DCL_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (max_batch <= 0 || max_seq <= 0) return fail(nullptr, DCL_ERR_INVALID_ARG, "max_batch/max_seq must be > 0");
  if (alloc && (!alloc->alloc || !alloc->free))
    return fail(nullptr, DCL_ERR_INVALID_ARG, "allocator needs alloc and free");
  if (cfg) {
    const dcl_model_config& m = *cfg;
    if (m.n_layers <= 0 || m.d_model <= 0 || m.n_heads <= 0 || m.n_kv_heads <= 0 || m.vocab <= 1 ||
        m.ffn_dim <= 0 || m.mask_id < 0 || m.mask_id >= m.vocab || !(m.rms_eps >= 0.f) || !(m.rope_theta > 0.f))
      return fail(nullptr, DCL_ERR_INVALID_ARG, "invalid model config");
    if ((m.head_dim != 64 && m.head_dim != 128) || m.d_model % 128 || m.ffn_dim % 128 ||
        m.n_heads % m.n_kv_heads || ((m.n_heads + m.n_kv_heads) * m.head_dim) % 128 ||
        (m.n_heads * m.head_dim) % 64 || m.vocab % 8)
      return fail(nullptr, DCL_ERR_UNSUPPORTED,
                  "unsupported shape (head_dim 64/128; d_model, ffn_dim multiples of 128; vocab multiple of 8)");
  }
  dcl_ctx* c = new dcl_ctx();
  c->max_batch = max_batch;
  c->max_seq = max_seq;
  c->stream = static_cast<cudaStream_t>(cuda_stream);
  if (!c->stream) {
    // a blocking stream: ordered with the legacy default stream, and capturable
    if (cudaStreamCreateWithFlags(&c->stream, cudaStreamDefault) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return fail(nullptr, DCL_ERR_CUDA, "stream creation failed (no CUDA device?)");
    }
    c->own_stream = true;
  }
  if (alloc) {
    c->alloc = *alloc;
    c->custom_alloc = true;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    release_stream(c);
    delete c;
    return fail(nullptr, DCL_ERR_CUDA, "no CUDA device");
  }
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10) {
    release_stream(c);
    delete c;
    return fail(nullptr, DCL_ERR_UNSUPPORTED, "needs a Blackwell (sm_10x) GPU, found sm_%d%d", major, minor);
  }
  c->derr = static_cast<int*>(dev_alloc(c, sizeof(int) * 4));
  if (!c->derr || cudaMemset(c->derr, 0, sizeof(int) * 4) != cudaSuccess) {
    dev_free_all(c);
    release_stream(c);
    delete c;
    return fail(nullptr, DCL_ERR_OOM, "device allocation failed");
  }
  if (cfg) {
    c->has_model = true;
    c->cfg = *cfg;
    const dcl_model_config& m = c->cfg;
    const size_t d = m.d_model, hd = m.head_dim, H = m.n_heads, G = m.n_kv_heads, F = m.ffn_dim, V = m.vocab;
    const size_t A = 128;  // elements (256 bytes)
    size_t off = 0;
    auto take = [&](size_t n) {
      const size_t o = off;
      off = align_up(off + n, A);
      return o;
    };
    const size_t o_embed = take(V * d), o_fn = take(d), o_lm = take(V * d);
    std::vector<size_t> lo(6 * m.n_layers);
    for (int l = 0; l < m.n_layers; ++l) {
      lo[6 * l + 0] = take(d);
      lo[6 * l + 1] = take((H + 2 * G) * hd * d);
      lo[6 * l + 2] = take(d * H * hd);
      lo[6 * l + 3] = take(d);
      lo[6 * l + 4] = take(2 * F * d);
      lo[6 * l + 5] = take(d * F);
    }
    c->wbuf = dev_alloc(c, off * sizeof(__nv_bfloat16));
    const size_t R = (size_t)max_batch * max_seq;
    const int nblk = gemm_lmhead_blocks(m.vocab);
    c->h = (float*)dev_alloc(c, sizeof(float) * R * d);
    c->xn = (__nv_bfloat16*)dev_alloc(c, 2 * R * d);
    c->qkv = (__nv_bfloat16*)dev_alloc(c, 2 * R * (H + 2 * G) * hd);
    c->attn = (__nv_bfloat16*)dev_alloc(c, 2 * R * H * hd);
    c->vt = (__half*)dev_alloc(c, 2 * (size_t)max_batch * G * hd * attn_vt_pitch(max_seq));
    c->kbuf = (__nv_bfloat16*)dev_alloc(c, 2 * R * G * hd);
    c->rp_buf = (int*)dev_alloc(c, sizeof(int) * (2 + 4 * R + 4 * (size_t)max_batch));
    c->act = (__nv_bfloat16*)dev_alloc(c, 2 * R * F);
    c->xg = (__nv_bfloat16*)dev_alloc(c, 2 * R * d);
    c->part = (float4*)dev_alloc(c, sizeof(float4) * R * nblk);
    c->ent_part = (float*)dev_alloc(c, sizeof(float) * R * nblk);
    c->ent = (float*)dev_alloc(c, 4 * R);
    c->conf = (float*)dev_alloc(c, 4 * R);
    c->jpde = (float*)dev_alloc(c, 4 * (size_t)max_batch);
    c->top1 = (int32_t*)dev_alloc(c, 4 * R);
    c->p1 = (float*)dev_alloc(c, 4 * R);
    c->p2 = (float*)dev_alloc(c, 4 * R);
    c->x = (int32_t*)dev_alloc(c, 4 * R);
    c->p = (int32_t*)dev_alloc(c, 4 * max_batch);
    c->k = (int32_t*)dev_alloc(c, 4 * max_batch);
    c->steps = (int32_t*)dev_alloc(c, 4 * max_batch);
    c->done_count = (int32_t*)dev_alloc(c, 16);
    c->x_init = (int32_t*)dev_alloc(c, 4 * R);
    c->p_init = (int32_t*)dev_alloc(c, 4 * max_batch);
    c->cmt = (uint8_t*)dev_alloc(c, R);
    c->cmt_init = (uint8_t*)dev_alloc(c, R);
    c->rope_cos = (float*)dev_alloc(c, 4 * (size_t)max_seq * hd / 2);
    c->rope_sin = (float*)dev_alloc(c, 4 * (size_t)max_seq * hd / 2);
    if (!c->wbuf || !c->h || !c->xn || !c->qkv || !c->attn || !c->vt || !c->kbuf || !c->rp_buf || !c->act || !c->xg || !c->part || !c->ent_part ||
        !c->ent || !c->conf || !c->jpde || !c->top1 ||
        !c->p1 || !c->p2 || !c->x || !c->p || !c->k || !c->steps || !c->done_count || !c->x_init || !c->p_init || !c->cmt || !c->cmt_init || !c->rope_cos ||
        !c->rope_sin) {
      dev_free_all(c);
      release_stream(c);
      delete c;
      return fail(nullptr, DCL_ERR_OOM, "device allocation of %.2f GB of weights + activations failed",
                  off * 2.0 / 1e9);
    }
    auto W = static_cast<__nv_bfloat16*>(c->wbuf);
    c->embed = W + o_embed;
    c->final_norm = W + o_fn;
    c->lm_head = W + o_lm;
    c->layers.resize(m.n_layers);
    for (int l = 0; l < m.n_layers; ++l)
      c->layers[l] = {W + lo[6 * l], W + lo[6 * l + 1], W + lo[6 * l + 2], W + lo[6 * l + 3], W + lo[6 * l + 4],
                      W + lo[6 * l + 5]};
    int* q = c->rp_buf;
    c->rp.counts = q;
    c->rp.row_seq = q + 2;
    c->rp.row_pos = c->rp.row_seq + R;
    c->rp.lm_src = c->rp.row_pos + R;
    c->rp.lm_slot = c->rp.lm_src + R;
    c->rp.seq_off = c->rp.lm_slot + R;
    c->rp.seq_len = c->rp.seq_off + max_batch;
    c->rp.pe_cache = c->rp.seq_len + max_batch;
    c->rp.kcap = c->rp.pe_cache + max_batch;
    if (rope_table_build(c->rope_cos, c->rope_sin, max_seq, (int)hd, m.rope_theta, c->stream) != cudaSuccess) {
      dev_free_all(c);
      release_stream(c);
      delete c;
      return fail(nullptr, DCL_ERR_CUDA, "RoPE table upload failed");
    }
  }
  if (cudaMallocHost(&c->h_done, 2 * sizeof(int32_t)) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->ev_done[0], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->ev_done[1], cudaEventDisableTiming) != cudaSuccess) {
    dev_free_all(c);
    release_stream(c);
    delete c;
    return fail(nullptr, DCL_ERR_CUDA, "pinned host buffer / event creation failed");
  }
  *out = c;
  return DCL_OK;
}

void dcl_destroy(dcl_ctx* c) {
  if (!c) return;
  if (c->stream) cudaStreamSynchronize(c->stream);
  if (c->gexec) cudaGraphExecDestroy(c->gexec);
  for (auto& l : c->launches) {
    cudaEventDestroy(l.start);
    cudaEventDestroy(l.stop);
  }
  if (c->ev_done[0]) cudaEventDestroy(c->ev_done[0]);
  if (c->ev_done[1]) cudaEventDestroy(c->ev_done[1]);
  if (c->h_done) cudaFreeHost(c->h_done);
  dev_free_all(c);
  release_stream(c);
  delete c;
}

dcl_status dcl_set_weight(dcl_ctx* c, int32_t kind, int32_t layer, const void* src, int32_t src_is_device) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->has_model) return fail(c, DCL_ERR_STATE, "ops-only context has no weights");
  if (!src) return fail(c, DCL_ERR_INVALID_ARG, "src is NULL");
  WDst w;
  if (!weight_dst(c, kind, layer, &w)) return fail(c, DCL_ERR_INVALID_ARG, "bad weight kind %d / layer %d", kind, layer);
  const cudaMemcpyKind mk = src_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  const size_t row_bytes = (size_t)w.cols * 2;
  if (w.blk_off < 0) {
    CUDA_TRY(c, cudaMemcpyAsync(w.ptr, src, row_bytes * w.rows, mk, c->stream));
  } else {  // 128-row blocks of gate (or up) go to the first (second) half of each 256-row group
    CUDA_TRY(c, cudaMemcpy2DAsync(w.ptr + (size_t)w.blk_off * w.cols, 256 * row_bytes, src, 128 * row_bytes,
                                  128 * row_bytes, (size_t)(w.rows / 128), mk, c->stream));
  }
  if (!src_is_device) CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  return DCL_OK;
}

dcl_status dcl_init_random_weights(dcl_ctx* c, uint64_t seed, float std, float lm_head_scale, float norm_gain_std) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->has_model) return fail(c, DCL_ERR_STATE, "ops-only context has no weights");
  if (seed >= 65536) return fail(c, DCL_ERR_INVALID_ARG, "seed must be < 65536");
  const float lm_std = std * lm_head_scale;
  for (int kind = 0; kind <= DCL_W_LM_HEAD; ++kind) {
    const bool global = kind == DCL_W_EMBED || kind == DCL_W_FINAL_NORM || kind == DCL_W_LM_HEAD;
    const bool norm = kind == DCL_W_ATTN_NORM || kind == DCL_W_MLP_NORM || kind == DCL_W_FINAL_NORM;
    for (int l = 0; l < (global ? 1 : c->cfg.n_layers); ++l) {
      WDst w;
      weight_dst(c, kind, l, &w);
      const float s = norm ? norm_gain_std : (kind == DCL_W_LM_HEAD ? lm_std : std);
      const float mean = norm ? 1.0f : 0.0f;
      const int64_t n = w.rows * w.cols;
      cudaError_t e = (w.blk_off < 0)
                          ? generate_launch(w.ptr, seed, tensor_id(kind, l), 0, n, s, mean, w.cols, 0, 0, 0, c->stream)
                          : generate_launch(w.ptr, seed, tensor_id(kind, l), 0, n, s, mean, w.cols, 128, 256,
                                            w.blk_off, c->stream);
      if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "weight generator: %s", cudaGetErrorString(e));
    }
  }
  return DCL_OK;
}

dcl_status dcl_set_prompt(dcl_ctx* c, int32_t batch, const int32_t* prompt, int32_t n_prompt,
                          const dcl_decode_config* cfg) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->has_model) return fail(c, DCL_ERR_STATE, "ops-only context has no model");
  if (!prompt || !cfg) return fail(c, DCL_ERR_INVALID_ARG, "prompt/cfg is NULL");
  if (batch <= 0 || batch > c->max_batch) return fail(c, DCL_ERR_INVALID_ARG, "batch %d outside [1, %d]", batch, c->max_batch);
  if (n_prompt < 0 || cfg->gen_len <= 0 || n_prompt + cfg->gen_len > c->max_seq)
    return fail(c, DCL_ERR_INVALID_ARG, "N + M = %d + %d exceeds max_seq %d", n_prompt, cfg->gen_len, c->max_seq);
  if (cfg->kv_cache < 0 || cfg->kv_cache > 2) return fail(c, DCL_ERR_INVALID_ARG, "kv_cache must be 0, 1 or 2");
  if (cfg->confidence != 0 && cfg->confidence != 1) return fail(c, DCL_ERR_INVALID_ARG, "confidence must be 0 or 1");
  if (cfg->acceptance != 0 && cfg->acceptance != 1) return fail(c, DCL_ERR_INVALID_ARG, "acceptance must be 0 or 1");
  if (cfg->acceptance == 1 && cfg->block_len <= 0)
    return fail(c, DCL_ERR_INVALID_ARG, "the threshold rule (acceptance = 1) needs block_len >= 1");
  if (cfg->kv_cache == 2 && cfg->acceptance != 0)
    return fail(c, DCL_ERR_UNSUPPORTED, "the dual cache (kv_cache = 2) is defined for the DCV acceptance");
  if (cfg->kv_cache && (cfg->block_len <= 0 || cfg->block_len % 32 || n_prompt % 32 || cfg->gen_len % 32))
    return fail(c, DCL_ERR_UNSUPPORTED, "the key / value cache needs N, M and the block length multiples of 32");
  if (cfg->max_window < 0 || cfg->min_commit < 0 || !(cfg->tau_commit == cfg->tau_commit) ||
      !(cfg->tau_draft == cfg->tau_draft))
    return fail(c, DCL_ERR_INVALID_ARG, "bad decode config");
  dcl_status s = validate_ids(c, prompt, (size_t)batch * n_prompt);
  if (s != DCL_OK) return s;
  const bool reshape = !c->prompt_set || batch != c->B || n_prompt != c->N || cfg->gen_len != c->M ||
                       cfg->kv_cache != c->dcfg.kv_cache;
  const int window = cfg->max_window > 0 ? cfg->max_window : (cfg->gen_len / 2 > 0 ? cfg->gen_len / 2 : 1);
  const bool redcv = !c->prompt_set || window != c->window || memcmp(cfg, &c->dcfg, sizeof *cfg) != 0;
  c->B = batch;
  c->N = n_prompt;
  c->M = cfg->gen_len;
  c->T = n_prompt + cfg->gen_len;
  c->window = window;
  c->dcfg = *cfg;
  std::vector<int32_t> xh((size_t)batch * c->T, c->cfg.mask_id), ph(batch, n_prompt), zero(batch, 0);
  std::vector<uint8_t> ch((size_t)batch * c->T, 0);
  for (int b = 0; b < batch; ++b) {
    memcpy(&xh[(size_t)b * c->T], prompt + (size_t)b * n_prompt, sizeof(int32_t) * n_prompt);
    memset(&ch[(size_t)b * c->T], 1, n_prompt);
  }
  CUDA_TRY(c, cudaMemcpyAsync(c->x, xh.data(), 4 * xh.size(), cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->p, ph.data(), 4 * batch, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->steps, zero.data(), 4 * batch, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->k, zero.data(), 4 * batch, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->x_init, c->x, 4 * xh.size(), cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->p_init, c->p, 4 * batch, cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->cmt, ch.data(), ch.size(), cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->cmt_init, c->cmt, ch.size(), cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->rp.pe_cache, 0xff, 4 * (size_t)batch, c->stream));  // no stored keys / values
  CUDA_TRY(c, cudaMemsetAsync(c->jpde, 0, 4 * (size_t)batch, c->stream));
  s = reset_done_count(c, ph.data());
  if (s != DCL_OK) return s;
  if (reshape) {
    c->prompt_set = false;
    s = build_plans(c);
    if (s != DCL_OK) return s;
  }
  if (reshape || redcv || !c->gexec) {
    s = build_graph(c);
    if (s != DCL_OK) return s;
  }
  c->prompt_set = true;
  return DCL_OK;
}

dcl_status dcl_step(dcl_ctx* c, int32_t* k_out) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "dcl_step before dcl_set_prompt");
  CUDA_TRY(c, cudaGraphLaunch(c->gexec, c->stream));
  c->profiled_step = c->profiling;
  if (k_out) {
    CUDA_TRY(c, cudaMemcpyAsync(k_out, c->k, 4 * c->B, cudaMemcpyDeviceToHost, c->stream));
    return check_device(c);
  }
  return DCL_OK;
}

dcl_status dcl_generate(dcl_ctx* c, int32_t max_steps, int32_t* out, dcl_stats* st) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "dcl_generate before dcl_set_prompt");
  if (max_steps < 0) return fail(c, DCL_ERR_INVALID_ARG, "max_steps < 0");
  const auto t0 = std::chrono::steady_clock::now();
  int launched = 0;
  bool done = false;
  // keep one step in flight: launch step s+1 before reading step s's finished-row count
  CUDA_TRY(c, cudaMemcpyAsync(&c->h_done[0], c->done_count, 4, cudaMemcpyDeviceToHost, c->stream));
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  done = c->h_done[0] >= c->B;
  while (!done && launched < max_steps) {
    CUDA_TRY(c, cudaGraphLaunch(c->gexec, c->stream));
    const int slot = launched & 1;
    CUDA_TRY(c, cudaMemcpyAsync(&c->h_done[slot], c->done_count, 4, cudaMemcpyDeviceToHost, c->stream));
    CUDA_TRY(c, cudaEventRecord(c->ev_done[slot], c->stream));
    ++launched;
    if (launched >= 2) {
      CUDA_TRY(c, cudaEventSynchronize(c->ev_done[slot ^ 1]));
      if (c->h_done[slot ^ 1] >= c->B) done = true;
    }
  }
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  if (launched > 0 && c->h_done[(launched - 1) & 1] >= c->B) done = true;
  c->profiled_step = c->profiling && launched > 0;
  dcl_status s = check_device(c);
  if (s != DCL_OK) return s;
  std::vector<int32_t> ph(c->B), sh(c->B);
  std::vector<float> jh(c->B);
  CUDA_TRY(c, cudaMemcpy(ph.data(), c->p, 4 * c->B, cudaMemcpyDeviceToHost));
  CUDA_TRY(c, cudaMemcpy(sh.data(), c->steps, 4 * c->B, cudaMemcpyDeviceToHost));
  CUDA_TRY(c, cudaMemcpy(jh.data(), c->jpde, 4 * c->B, cudaMemcpyDeviceToHost));
  if (out) {
    for (int b = 0; b < c->B; ++b)
      CUDA_TRY(c, cudaMemcpy(out + (size_t)b * c->M, c->x + (size_t)b * c->T + c->N, 4 * c->M,
                             cudaMemcpyDeviceToHost));
  }
  const double ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
  if (st) {
    int64_t tok = 0, stp = 0;
    double jp = 0.0;
    for (int b = 0; b < c->B; ++b) {
      tok += ph[b] - c->N;
      stp = sh[b] > stp ? sh[b] : stp;
      jp += jh[b];
    }
    st->jpde_bound = jp;
    st->steps = stp;
    st->tokens = tok;
    st->elapsed_ms = ms;
    st->done = done ? 1 : 0;
  }
  if (!done) return fail(c, DCL_ERR_TIMEOUT, "max_steps = %d reached before every row finished", max_steps);
  return DCL_OK;
}

dcl_status dcl_restart(dcl_ctx* c) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "no prompt set");
  const size_t B = c->B;
  CUDA_TRY(c, cudaMemcpyAsync(c->x, c->x_init, 4 * B * c->T, cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->p, c->p_init, 4 * B, cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->cmt, c->cmt_init, B * c->T, cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->steps, 0, 4 * B, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->k, 0, 4 * B, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->done_count, 0, 4, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->rp.pe_cache, 0xff, 4 * B, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->jpde, 0, 4 * B, c->stream));
  return DCL_OK;
}

dcl_status dcl_get_state(dcl_ctx* c, int32_t* x, int32_t* p) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "no prompt set");
  if (x) CUDA_TRY(c, cudaMemcpyAsync(x, c->x, 4 * (size_t)c->B * c->T, cudaMemcpyDeviceToHost, c->stream));
  if (p) CUDA_TRY(c, cudaMemcpyAsync(p, c->p, 4 * (size_t)c->B, cudaMemcpyDeviceToHost, c->stream));
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  return DCL_OK;
}

dcl_status dcl_set_state(dcl_ctx* c, const int32_t* x, const int32_t* p) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "no prompt set");
  if (!x || !p) return fail(c, DCL_ERR_INVALID_ARG, "x/p is NULL");
  dcl_status s = validate_ids(c, x, (size_t)c->B * c->T);
  if (s != DCL_OK) return s;
  for (int b = 0; b < c->B; ++b)
    if (p[b] < c->N || p[b] > c->T) return fail(c, DCL_ERR_INVALID_ARG, "p[%d] = %d outside [N, N+M]", b, p[b]);
  // committed flags (read by the threshold rule only): every position before p, and every
  // later position that holds a token other than MASK
  std::vector<uint8_t> ch((size_t)c->B * c->T);
  for (int b = 0; b < c->B; ++b)
    for (int i = 0; i < c->T; ++i)
      ch[(size_t)b * c->T + i] = (i < p[b] || x[(size_t)b * c->T + i] != c->cfg.mask_id) ? 1 : 0;
  CUDA_TRY(c, cudaMemcpyAsync(c->cmt, ch.data(), ch.size(), cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->x, x, 4 * (size_t)c->B * c->T, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemcpyAsync(c->p, p, 4 * (size_t)c->B, cudaMemcpyHostToDevice, c->stream));
  CUDA_TRY(c, cudaMemsetAsync(c->rp.pe_cache, 0xff, 4 * (size_t)c->B, c->stream));  // the next step refreshes
  CUDA_TRY(c, cudaMemsetAsync(c->jpde, 0, 4 * (size_t)c->B, c->stream));
  return reset_done_count(c, p);
}

namespace {
// The parity hooks' common body: the forward (from the embedding, or from block `layer` on
// h_in), optionally the acceptance, then copies of the predictions.
dcl_status forward_debug_impl(dcl_ctx* c, int layer, const float* h_in, bool commit, void* logits_dev,
                              int32_t* top1_dev, float* p1_dev, float* p2_dev, float* conf_dev, float* entropy_dev) {
  const size_t R = (size_t)c->B * c->T;
  if (!c->snap || c->snap_rows < R) {
    c->snap = (float*)dev_alloc(c, sizeof(float) * (c->cfg.n_layers + 1) * R * c->cfg.d_model);
    if (!c->snap) return fail(c, DCL_ERR_OOM, "snapshot buffer allocation failed");
    c->snap_rows = R;
  }
  const char* what = nullptr;
  cudaError_t e = enqueue_step(c, commit, false, true, &what, layer, h_in);
  if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "forward failed at %s: %s", what ? what : "?", cudaGetErrorString(e));
  const size_t G = (size_t)c->B * c->M;
  if (top1_dev) CUDA_TRY(c, cudaMemcpyAsync(top1_dev, c->top1, 4 * G, cudaMemcpyDeviceToDevice, c->stream));
  if (p1_dev) CUDA_TRY(c, cudaMemcpyAsync(p1_dev, c->p1, 4 * G, cudaMemcpyDeviceToDevice, c->stream));
  if (p2_dev) CUDA_TRY(c, cudaMemcpyAsync(p2_dev, c->p2, 4 * G, cudaMemcpyDeviceToDevice, c->stream));
  if (conf_dev)
    CUDA_TRY(c, cudaMemcpyAsync(conf_dev, c->dcfg.confidence ? c->conf : c->p1, 4 * G, cudaMemcpyDeviceToDevice,
                                c->stream));
  if (entropy_dev) CUDA_TRY(c, cudaMemcpyAsync(entropy_dev, c->ent, 4 * G, cudaMemcpyDeviceToDevice, c->stream));
  if (logits_dev) {
    GemmPlan pl;
    EpiParams ep;
    ep.out = logits_dev;
    ep.ldo = c->cfg.vocab;
    const char* why = nullptr;
    if (gemm_plan(&pl, c->xg, (int)G, c->cfg.d_model, c->lm_head, c->cfg.vocab, EPI_BF16, ep, c->num_sms, 0, &why))
      return fail(c, DCL_ERR_UNSUPPORTED, "logits plan: %s", why ? why : "?");
    dcl_status s = attach_scratch(c, &pl);
    if (s != DCL_OK) return s;
    const cudaError_t e = gemm_launch(pl, c->derr, c->stream);
    release_scratch(c, &pl);
    if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "logits GEMM: %s", cudaGetErrorString(e));
  }
  return check_device(c);
}
}  // namespace

dcl_status dcl_forward_debug(dcl_ctx* c, void* logits_dev, int32_t* top1_dev, float* p1_dev, float* p2_dev,
                             float* conf_dev, float* entropy_dev) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "no prompt set");
  return forward_debug_impl(c, 0, nullptr, false, logits_dev, top1_dev, p1_dev, p2_dev, conf_dev, entropy_dev);
}

dcl_status dcl_forward_debug_from(dcl_ctx* c, int32_t layer, const float* h_dev, int32_t commit, void* logits_dev,
                                  int32_t* top1_dev, float* p1_dev, float* p2_dev, float* conf_dev,
                                  float* entropy_dev) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set) return fail(c, DCL_ERR_STATE, "no prompt set");
  if (!h_dev || layer < 0 || layer > c->cfg.n_layers || (commit != 0 && commit != 1))
    return fail(c, DCL_ERR_INVALID_ARG, "bad layer / h / commit");
  if (c->dcfg.kv_cache) return fail(c, DCL_ERR_UNSUPPORTED, "a forward from a given stream needs full recompute");
  // the stream's rows are every (sequence, position): no sequence may have finished (a
  // finished sequence contributes no rows to the step)
  std::vector<int32_t> ph(c->B);
  CUDA_TRY(c, cudaMemcpyAsync(ph.data(), c->p, 4 * (size_t)c->B, cudaMemcpyDeviceToHost, c->stream));
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  for (int b = 0; b < c->B; ++b)
    if (ph[b] >= c->T) return fail(c, DCL_ERR_STATE, "sequence %d has finished", b);
  return forward_debug_impl(c, layer, h_dev, commit != 0, logits_dev, top1_dev, p1_dev, p2_dev, conf_dev,
                            entropy_dev);
}

dcl_status dcl_debug_hidden(dcl_ctx* c, int32_t layer, float* h_dev) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->prompt_set || !c->snap) return fail(c, DCL_ERR_STATE, "call dcl_forward_debug first");
  if (layer < -1 || layer >= c->cfg.n_layers || !h_dev) return fail(c, DCL_ERR_INVALID_ARG, "bad layer / pointer");
  const size_t n = (size_t)c->B * c->T * c->cfg.d_model;
  CUDA_TRY(c, cudaMemcpyAsync(h_dev, c->snap + (size_t)(layer + 1) * n, sizeof(float) * n,
                              cudaMemcpyDeviceToDevice, c->stream));
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  return DCL_OK;
}

dcl_status dcl_accept(dcl_ctx* c, const void* logits_dev, int32_t B, int32_t P, int32_t V,
                      const int32_t* committed_dev, int32_t* x_dev, const dcl_decode_config* cfg, int32_t* k_dev) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!logits_dev || !committed_dev || !x_dev || !cfg || !k_dev) return fail(c, DCL_ERR_INVALID_ARG, "NULL argument");
  if (B <= 0 || P <= 0 || V <= 1 || P > 4096 || (int64_t)B * P > (1 << 20))
    return fail(c, DCL_ERR_INVALID_ARG, "bad B/P/V (P <= 4096, B*P <= 2^20)");
  if (cfg->max_window < 0 || cfg->min_commit < 0 || (cfg->confidence != 0 && cfg->confidence != 1) ||
      (cfg->acceptance != 0 && cfg->acceptance != 1))
    return fail(c, DCL_ERR_INVALID_ARG, "bad decode config");
  const size_t n = (size_t)B * P;
  if (c->acc_cap < n) {
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));  // no launch may still use the old buffers
    dev_free_one(c, c->acc_ids);
    dev_free_one(c, c->acc_c1);
    dev_free_one(c, c->acc_c2);
    c->acc_cap = 0;
    c->acc_ids = (int32_t*)dev_alloc(c, 4 * n);
    c->acc_c1 = (float*)dev_alloc(c, 4 * n);
    c->acc_c2 = (float*)dev_alloc(c, 4 * n);
    if (!c->acc_ids || !c->acc_c1 || !c->acc_c2) return fail(c, DCL_ERR_OOM, "accept scratch allocation failed");
    c->acc_cap = n;
  }
  const int window = cfg->max_window > 0 ? cfg->max_window : (P / 2 > 0 ? P / 2 : 1);
  DcvParams prm{cfg->tau_commit, cfg->tau_draft, window, cfg->min_commit, cfg->contiguous_drafts,
                cfg->acceptance, P};
  CUDA_TRY(c, accept_stats_launch(static_cast<const __nv_bfloat16*>(logits_dev), committed_dev, B, P, V, c->acc_ids,
                                  c->acc_c1, c->acc_c2, cfg->confidence, c->stream));
  CUDA_TRY(c, accept_commit_launch(committed_dev, c->acc_ids, c->acc_c1, x_dev, k_dev, B, P, prm, c->stream));
  return DCL_OK;
}

dcl_status dcl_op_rmsnorm(dcl_ctx* c, const float* x_dev, const void* gain_dev, void* y_dev, int32_t rows, int32_t d,
                          float eps) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!x_dev || !gain_dev || !y_dev || rows <= 0 || d <= 0 || d % 4) return fail(c, DCL_ERR_INVALID_ARG, "bad rmsnorm args");
  CUDA_TRY(c, rmsnorm_launch(x_dev, static_cast<const __nv_bfloat16*>(gain_dev), static_cast<__nv_bfloat16*>(y_dev),
                             rows, d, eps, nullptr, nullptr, c->stream));
  return DCL_OK;
}

dcl_status dcl_op_linear(dcl_ctx* c, const void* a_dev, const void* w_dev, void* out_dev, int32_t M, int32_t N,
                         int32_t K, int32_t mode, int32_t tile) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!a_dev || !w_dev || !out_dev || (mode != 0 && mode != 1)) return fail(c, DCL_ERR_INVALID_ARG, "bad linear args");
  if (tile != 0 && tile != 128 && tile != 256 && (tile & 0xff) != kTilePair)
    return fail(c, DCL_ERR_INVALID_ARG, "bad tile");
  GemmPlan pl;
  EpiParams ep;
  ep.out = out_dev;
  ep.ldo = N;
  const char* why = nullptr;
  if (gemm_plan(&pl, a_dev, M, K, w_dev, N, mode == 0 ? EPI_BF16 : EPI_RESID_F32, ep, c->num_sms, tile, &why))
    return fail(c, DCL_ERR_INVALID_ARG, "%s", why ? why : "bad GEMM shape");
  dcl_status s = attach_scratch(c, &pl);
  if (s != DCL_OK) return s;
  const cudaError_t e = gemm_launch(pl, c->derr, c->stream);
  release_scratch(c, &pl);
  if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "GEMM launch: %s", cudaGetErrorString(e));
  return check_device(c);
}

dcl_status dcl_op_attention(dcl_ctx* c, const void* qkv_dev, void* out_dev, int32_t batch, int32_t T, int32_t H,
                            int32_t G, int32_t hd, int32_t q_rows) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!qkv_dev || !out_dev || batch <= 0 || T <= 0 || H <= 0 || G <= 0 || H % G || (hd != 64 && hd != 128) ||
      q_rows < 0 || q_rows > T || q_rows % 32)
    return fail(c, DCL_ERR_INVALID_ARG, "bad attention args");
  __half* vt = static_cast<__half*>(dev_alloc(c, 2 * (size_t)batch * G * hd * attn_vt_pitch(T)));
  int* tab = q_rows > 0 ? static_cast<int*>(dev_alloc(c, sizeof(int) * 2 * (size_t)batch)) : nullptr;
  auto release = [&]() {
    cudaStreamSynchronize(c->stream);
    dev_free_one(c, vt);
    dev_free_one(c, tab);
  };
  if (!vt || (q_rows > 0 && !tab)) {
    release();
    return fail(c, DCL_ERR_OOM, "attention scratch allocation failed");
  }
  if (tab) {  // sequence b's queries: positions [T - q_rows, T), rows b*T + T - q_rows onwards
    std::vector<int> th(2 * (size_t)batch);
    for (int b = 0; b < batch; ++b) {
      th[b] = b * T + T - q_rows;
      th[batch + b] = q_rows;
    }
    CUDA_TRY(c, cudaMemcpyAsync(tab, th.data(), sizeof(int) * th.size(), cudaMemcpyHostToDevice, c->stream));
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  }
  AttnPlan pl;
  if (attention_plan(&pl, static_cast<const __nv_bfloat16*>(qkv_dev), nullptr, vt, static_cast<__nv_bfloat16*>(out_dev),
                     batch, T, H, G, hd, batch * T, tab, tab ? tab + batch : nullptr) != cudaSuccess) {
    release();
    return fail(c, DCL_ERR_INVALID_ARG, "attention: operands must be 16-byte aligned");
  }
  const cudaError_t e = attention_launch(pl, c->derr, c->stream);
  if (e != cudaSuccess) {
    release();
    return fail(c, DCL_ERR_CUDA, "attention launch: %s", cudaGetErrorString(e));
  }
  const dcl_status s = check_device(c);
  release();
  return s;
}

dcl_status dcl_op_lmhead_top2(dcl_ctx* c, const void* x_dev, const void* w_dev, int32_t R, int32_t V, int32_t d,
                              int32_t* top1_dev, float* p1_dev, float* p2_dev, float* entropy_dev, int32_t tile) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!x_dev || !w_dev || !top1_dev || !p1_dev || !p2_dev || R <= 0 || V <= 1)
    return fail(c, DCL_ERR_INVALID_ARG, "bad lmhead args");
  if (tile != 0 && tile != 256 && (tile & 0xff) != kTilePair) return fail(c, DCL_ERR_INVALID_ARG, "bad tile");
  const int nblk = gemm_lmhead_blocks(V);
  // {max, sum, id, second} partials, then (with entropy_dev) the entropy partials
  float4* part = static_cast<float4*>(dev_alloc(c, (sizeof(float4) + (entropy_dev ? 4 : 0)) * (size_t)R * nblk));
  if (!part) return fail(c, DCL_ERR_OOM, "partials allocation failed");
  float* upart = entropy_dev ? reinterpret_cast<float*>(part + (size_t)R * nblk) : nullptr;
  GemmPlan pl;
  EpiParams ep;
  ep.out = part;
  ep.ent_part = upart;
  const char* why = nullptr;
  if (gemm_plan(&pl, x_dev, R, d, w_dev, V, EPI_LMHEAD, ep, c->num_sms, tile, &why)) {
    dev_free_one(c, part);
    return fail(c, DCL_ERR_INVALID_ARG, "%s", why ? why : "bad LM-head shape");
  }
  dcl_status s = attach_scratch(c, &pl);
  if (s != DCL_OK) {
    dev_free_one(c, part);
    return s;
  }
  const cudaError_t e = gemm_launch(pl, c->derr, c->stream);
  release_scratch(c, &pl);
  if (e != cudaSuccess) {
    dev_free_one(c, part);
    return fail(c, DCL_ERR_CUDA, "LM-head GEMM: %s", cudaGetErrorString(e));
  }
  ConfOut co;
  co.top1 = top1_dev;
  co.p1 = p1_dev;
  co.p2 = p2_dev;
  co.ent = entropy_dev;
  CUDA_TRY(c, lmhead_combine_launch(part, upart, R, nblk, co, nullptr, nullptr, c->stream));
  s = check_device(c);
  dev_free_one(c, part);
  return s;
}

dcl_status dcl_op_generate(dcl_ctx* c, void* dst_dev, uint64_t seed, int32_t tid, int64_t start, int64_t count,
                           float std, float mean) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!dst_dev || seed >= 65536 || tid < 0 || tid >= 65536 || start < 0 || count < 0 || start + count > (1ll << 32))
    return fail(c, DCL_ERR_INVALID_ARG, "bad generator args");
  CUDA_TRY(c, generate_launch(static_cast<__nv_bfloat16*>(dst_dev), seed, tid, start, count, std, mean, 1, 0, 0, 0,
                              c->stream));
  return DCL_OK;
}

dcl_status dcl_selftest_wait_timeout(dcl_ctx* c, int32_t which) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (which != 0 && which != 1) return fail(c, DCL_ERR_INVALID_ARG, "which must be 0 or 1");
  int* flag = static_cast<int*>(dev_alloc(c, sizeof(int)));
  if (!flag) return fail(c, DCL_ERR_OOM, "flag allocation failed");
  cudaError_t e = cudaMemsetAsync(flag, 0, sizeof(int), c->stream);
  if (e == cudaSuccess) e = wait_selftest_launch(which, flag, c->derr, c->stream);
  if (e != cudaSuccess) {
    dev_free_one(c, flag);
    return fail(c, DCL_ERR_CUDA, "self-test launch: %s", cudaGetErrorString(e));
  }
  const dcl_status s = check_device(c);
  dev_free_one(c, flag);
  return s;
}

dcl_status dcl_launch_floor(dcl_ctx* c, int32_t n_kernels, int32_t reps, float* ms_per_graph) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (n_kernels < 1 || n_kernels > 100000 || reps < 1 || !ms_per_graph)
    return fail(c, DCL_ERR_INVALID_ARG, "need 1 <= n_kernels <= 100000, reps >= 1 and an output");
  cudaGraph_t g = nullptr;
  cudaGraphExec_t ge = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  cudaError_t e = cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal);
  for (int i = 0; i < n_kernels && e == cudaSuccess; ++i) e = empty_launch(c->stream);
  cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
  if (e == cudaSuccess) e = e2;
  if (e == cudaSuccess) e = cudaGraphInstantiate(&ge, g, 0);
  if (e == cudaSuccess) e = cudaEventCreate(&e0);
  if (e == cudaSuccess) e = cudaEventCreate(&e1);
  for (int i = 0; i < 3 && e == cudaSuccess; ++i) e = cudaGraphLaunch(ge, c->stream);  // warm-up
  if (e == cudaSuccess) e = cudaEventRecord(e0, c->stream);
  for (int i = 0; i < reps && e == cudaSuccess; ++i) e = cudaGraphLaunch(ge, c->stream);
  if (e == cudaSuccess) e = cudaEventRecord(e1, c->stream);
  if (e == cudaSuccess) e = cudaEventSynchronize(e1);
  float ms = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (ge) cudaGraphExecDestroy(ge);
  if (g) cudaGraphDestroy(g);
  if (e != cudaSuccess) return fail(c, DCL_ERR_CUDA, "launch floor: %s", cudaGetErrorString(e));
  *ms_per_graph = ms / reps;
  return DCL_OK;
}

dcl_status dcl_set_profiling(dcl_ctx* c, int32_t enable) {
  if (!c) return DCL_ERR_INVALID_ARG;
  c->profiling = enable != 0;
  if (c->prompt_set) return build_graph(c);
  return DCL_OK;
}

dcl_status dcl_profile_last_step(dcl_ctx* c, float* ms, int32_t* kind, int32_t cap, int32_t* n) {
  if (!c) return DCL_ERR_INVALID_ARG;
  if (!c->profiling || !c->profiled_step) return fail(c, DCL_ERR_STATE, "no profiled step has run");
  CUDA_TRY(c, cudaStreamSynchronize(c->stream));
  const int cnt = (int)c->launch_i;
  int w = 0;
  for (int i = 0; i < cnt && w < cap; ++i, ++w) {
    float t = 0.f;
    CUDA_TRY(c, cudaEventElapsedTime(&t, c->launches[i].start, c->launches[i].stop));
    if (ms) ms[w] = t;
    if (kind) kind[w] = c->launches[i].kind;
  }
  if (n) *n = w;
  return DCL_OK;
}

}  // extern "C"
