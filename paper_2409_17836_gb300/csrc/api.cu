// api.cu -- the C ABI of liblmgc.so (include/lmgc.h): context, model forward orchestration,
// the encode pipeline (Sec. 4: serialise -> windows from BOS -> LM -> integer CDF -> one
// arithmetic code per window -> container) and the KV-cached decode (Sec. 4 "Compression").
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <string>
#include <vector>

#include "lmgc_internal.cuh"

namespace lmgc {

static thread_local std::string g_thread_err;
static std::atomic<unsigned long long> g_launches{0};

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

void set_thread_error(const std::string& s) { g_thread_err = s; }

// tokens of n serialised values under the context's layout (Sec. 4; byte grouping, Sec. 5.3)
static int64_t n_tokens(const lmgc_ctx* ctx, int64_t n) {
  return serial_tokens(ctx->cfg.input_kind, ctx->cfg.sep_mode, ctx->cfg.byte_group, n);
}

lmgc_status fail(lmgc_ctx* ctx, lmgc_status st, const std::string& msg) {
  if (ctx) ctx->err = msg;
  g_thread_err = msg;
  return st;
}

lmgc_status cuda_fail(lmgc_ctx* ctx, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  return fail(ctx, e == cudaErrorMemoryAllocation ? LMGC_ERR_NOMEM : LMGC_ERR_CUDA, m);
}

// CRC-32 (IEEE 802.3, reflected 0xEDB88320), for the container header.
static uint32_t crc32(const uint8_t* p, size_t n) {
  static uint32_t table[256];
  static bool init = false;
  if (!init) {
    for (uint32_t i = 0; i < 256; i++) {
      uint32_t c = i;
      for (int k = 0; k < 8; k++) c = (c & 1u) ? (0xEDB88320u ^ (c >> 1)) : (c >> 1);
      table[i] = c;
    }
    init = true;
  }
  uint32_t c = 0xFFFFFFFFu;
  for (size_t i = 0; i < n; i++) c = table[(c ^ p[i]) & 0xFFu] ^ (c >> 8);
  return c ^ 0xFFFFFFFFu;
}

static uint32_t model_crc(const lmgc_config& c) {
  uint8_t b[40];
  int32_t iv[7] = {c.n_layers, c.d_model, c.n_heads, c.n_kv_heads, c.d_ffn, c.vocab, c.dtype == LMGC_BF16 ? 1 : 0};
  float fv[3] = {c.init_std, c.rms_eps, c.rope_theta};
  memcpy(b, iv, 28);
  memcpy(b + 28, fv, 12);
  return crc32(b, 40);
}

// ---- profiling of kernel classes (CUDA events around launches, only when enabled) ----
enum KClass { kGemm = 0, kAttn = 1, kCdf = 2, kCoder = 3, kSer = 4, kNorm = 5, kOther = 6, kNumClasses = 7 };
static const char* kClassNames[kNumClasses] = {"gemm", "attention", "cdf_pairs", "range_encode", "serialize",
                                                "norm_rope_act", "other"};

static cudaEvent_t prof_event(lmgc_ctx* ctx) {
  if (!ctx->prof.pool.empty()) {
    cudaEvent_t e = ctx->prof.pool.back();
    ctx->prof.pool.pop_back();
    return e;
  }
  cudaEvent_t e;
  cudaEventCreate(&e);
  return e;
}

// Context-free entry points (lmgc_range_encode) record into this process-wide context.
static lmgc_ctx* free_ctx() {
  static lmgc_ctx* c = [] {
    lmgc_ctx* x = new lmgc_ctx();
    for (int i = 0; i < kNumClasses; i++) x->prof.stats[i] = KernelStat{kClassNames[i], 0, 0.f, 0.0};
    return x;
  }();
  return c;
}

struct ProfScope {
  lmgc_ctx* ctx;
  cudaStream_t s;
  bool on;
  ProfScope(lmgc_ctx* c, int cls, double work, cudaStream_t st) : ctx(c ? c : free_ctx()), s(st) {
    on = ctx->prof.enabled;
    if (!on) return;
    Profiler::Rec r;
    r.cls = cls;
    r.work = work;
    r.a = prof_event(ctx);
    r.b = prof_event(ctx);
    cudaEventRecord(r.a, s);
    ctx->prof.pending.push_back(r);
  }
  ~ProfScope() {
    if (on) cudaEventRecord(ctx->prof.pending.back().b, s);
  }
};

static void prof_collect(lmgc_ctx* ctx) {
  for (auto& r : ctx->prof.pending) {
    float ms = 0.f;
    cudaEventSynchronize(r.b);
    cudaEventElapsedTime(&ms, r.a, r.b);
    KernelStat& st = ctx->prof.stats[r.cls];
    st.launches++;
    st.ms += ms;
    st.work += r.work;
    ctx->prof.pool.push_back(r.a);
    ctx->prof.pool.push_back(r.b);
  }
  ctx->prof.pending.clear();
}

// ---- GEMM dispatch by the model's dtype: a bf16-weight model runs every contraction on the
// fp16 tcgen05 kernel, an fp32 model on the three-pass TF32 tcgen05 kernel (lmgc_create rejects
// shapes and devices they do not take) ----
static void gemm(lmgc_ctx* ctx, const void* A, const void* B, void* C, int64_t M, int64_t N, int64_t K, int epi,
                 cudaStream_t s, const RopeArgs* rope = nullptr, const NormArgs* norm = nullptr) {
  ProfScope ps(ctx, kGemm, 2.0 * (double)M * (double)N * (double)K, s);
  if (ctx->cfg.dtype == LMGC_BF16)
    launch_gemm_tc(A, B, C, M, N, K, epi, ctx->d_err, s, rope, norm);
  else  // kSwiGLU and kQKVRope never reach here
    launch_gemm_tf32((const float*)A, (const float*)B, (float*)C, M, N, K, epi, ctx->d_err, s);
}

// kv: the qkv rows themselves (prefill), or the decoder's cache (from_cache), whose rows hold a
// position's keys and values only: [K heads | V heads], 2 n_kv_heads hd wide
static void attention(lmgc_ctx* ctx, const void* q, const void* kv, void* out, int64_t n_win, int64_t pos_first,
                      int n_pos, int64_t q_win_stride, cudaStream_t s, bool from_cache = false) {
  const lmgc_config& c = ctx->cfg;
  // algorithmic flops: QK^T and PV over the causal triangle, 4*hd per (query, key) pair per head
  double pairs = 0;
  for (int64_t p = pos_first; p < pos_first + n_pos; p++) pairs += (double)(p + 1);
  ProfScope ps(ctx, kAttn, 4.0 * ctx->hd * c.n_heads * pairs * (double)n_win, s);
  const int qd = c.n_heads * ctx->hd, kd = c.n_kv_heads * ctx->hd;
  const int64_t kv_dim = from_cache ? 2 * kd : ctx->qkv_dim;
  const int k_off = from_cache ? 0 : qd, v_off = k_off + kd;
  // lmgc_create admitted only head layouts the tcgen05 kernels take
  const int64_t q_rows = q_win_stride == 1 ? n_win : n_win * c.window;
  if (c.dtype == LMGC_BF16)
    launch_attention_tc(q, q_rows, ctx->qkv_dim, kv, n_win * c.window, kv_dim, k_off, v_off, out, qd, c.n_heads,
                        c.n_kv_heads, ctx->hd, c.window, n_win, pos_first, n_pos, q_win_stride, ctx->d_err, s);
  else
    launch_attention_tf32((const float*)q, q_rows, ctx->qkv_dim, (const float*)kv, n_win * c.window, kv_dim, k_off,
                          v_off, (float*)out, qd, c.n_heads, c.n_kv_heads, ctx->hd, c.window, n_win, pos_first,
                          n_pos, q_win_stride, ctx->d_err, s);
}

// One forward of the model over `rows` input rows already embedded into ws.x.
//   prefill: rows = n_win * W, row r at position r mod W, keys/values from ws.qkv itself
//   decode:  rows = n_win, every row at position pos; keys/values from the cache
// narrow: the vocabulary projection over the restricted alphabet's rows only (w_head_alpha,
// logits [rows][kAlphaCols]) instead of all V rows.
static void forward_layers(lmgc_ctx* ctx, int64_t rows, int64_t n_win, bool decode, int64_t pos, cudaStream_t s,
                           bool narrow = false) {
  const lmgc_config& c = ctx->cfg;
  const void* w_head = narrow ? ctx->w_head_alpha : ctx->w_head;
  const int64_t n_head = narrow ? kAlphaCols : c.vocab;
  const int d = c.d_model, F = c.d_ffn, hd = ctx->hd, qd = c.n_heads * hd;
  Workspace& ws = ctx->ws;
  const int64_t W = c.window;
  if (ctx->fused_norm) {
    // RMSNorm folded into the GEMMs: the residual producers (embedding, O and down projections)
    // leave x (fp32), fp16(x) in ws.n and per-256-column sums of squares in ws.ss; the consumers
    // (QKV, gate/up, vocabulary) read fp16(x) and scale each row by rsqrt(mean(x^2) + eps).
    __half* xh = (__half*)ws.n;
    const NormArgs consume{ws.ss, d / 256, 1.0f / (float)d, c.rms_eps, nullptr, nullptr};
    const NormArgs produce{nullptr, 0, 0.f, 0.f, xh, ws.ss};
    const bool wide_o = qd <= 2048;  // measured: +5% at K = 2048, -2% at K = 4096
    const NormArgs consume_o{ws.ss, d / 128, 1.0f / (float)d, c.rms_eps, nullptr, nullptr};
    for (int l = 0; l < c.n_layers; l++) {
      const Layer& L = ctx->layers[l];
      RopeArgs ra{ctx->rope_cs, (c.n_heads + c.n_kv_heads) * hd, hd, decode ? 1 : c.window, decode ? pos : 0};
      gemm(ctx, xh, L.wqkv, ws.qkv, rows, ctx->qkv_dim, d, kQKVRope, s, &ra, &consume);
      if (!decode) {
        attention(ctx, ws.qkv, ws.qkv, ws.att, n_win, 0, c.window, W, s);
      } else {
        // the cache keeps each position's keys and values (columns [qd, qd + 2 kd) of its qkv row)
        char* cache_l = (char*)ctx->kv_cache + (size_t)l * (size_t)n_win * W * ctx->kv_dim * ctx->elt;
        launch_copy_rows((const char*)ws.qkv + (size_t)qd * ctx->elt, ctx->qkv_dim, cache_l, W, pos, n_win,
                         ctx->kv_dim, c.dtype, s);
        attention(ctx, ws.qkv, cache_l, ws.att, n_win, pos, 1, 1, s, true);
      }
      // the O projection (K = qd, a short main loop) takes the 8-warp residual epilogue, whose
      // sums of squares come in 128-column parts; the choice depends on the shape only, so a
      // decode makes the same one
      gemm(ctx, ws.att, L.wo, ws.x, rows, d, qd, wide_o ? kAddResidualWide : kAddResidual, s, nullptr, &produce);
      gemm(ctx, xh, L.wgu, ws.act, rows, 2 * (int64_t)F, d, kSwiGLU, s, nullptr, wide_o ? &consume_o : &consume);
      gemm(ctx, ws.act, L.wdown, ws.x, rows, d, F, kAddResidual, s, nullptr, &produce);
    }
    // a prefill also leaves each logits row's maximum for the CDF kernel (the transposing fp32
    // epilogue, which takes vocabularies that are multiples of 32, computes it)
    NormArgs head = consume;
    const bool with_max = !decode && !narrow && c.vocab % 32 == 0;
    if (with_max) {
      cudaMemsetAsync(ctx->row_max, 0, (size_t)rows * 4, s);
      head.row_max = ctx->row_max;
    }
    gemm(ctx, xh, w_head, ctx->logits, rows, n_head, d, kStoreF32, s, nullptr, &head);
    ctx->row_max_valid = with_max;
    return;
  }
  for (int l = 0; l < c.n_layers; l++) {
    const Layer& L = ctx->layers[l];
    {
      ProfScope ps(ctx, kNorm, 0, s);
      launch_rmsnorm(ws.x, rows, d, c.rms_eps, ws.n, c.dtype, s);
    }
    if (ctx->fused_rope) {
      RopeArgs ra{ctx->rope_cs, (c.n_heads + c.n_kv_heads) * hd, hd, decode ? 1 : c.window, decode ? pos : 0};
      ProfScope ps(ctx, kGemm, 2.0 * (double)rows * (double)ctx->qkv_dim * (double)d, s);
      launch_gemm_tc(ws.n, L.wqkv, ws.qkv, rows, ctx->qkv_dim, d, kQKVRope, ctx->d_err, s, &ra);
    } else {
      gemm(ctx, ws.n, L.wqkv, ws.qkv, rows, ctx->qkv_dim, d, kStore, s);
      ProfScope ps(ctx, kNorm, 0, s);
      launch_rope(ws.qkv, rows, ctx->qkv_dim, c.n_heads + c.n_kv_heads, hd, ctx->rope_cs, c.window,
                  decode ? pos : 0, decode ? 1 : W, decode ? 1 : c.window, c.dtype, s);
    }
    if (!decode) {
      attention(ctx, ws.qkv, ws.qkv, ws.att, n_win, 0, c.window, W, s);
    } else {
      char* cache_l = (char*)ctx->kv_cache + (size_t)l * (size_t)n_win * W * ctx->kv_dim * ctx->elt;
      launch_copy_rows((const char*)ws.qkv + (size_t)qd * ctx->elt, ctx->qkv_dim, cache_l, W, pos, n_win,
                       ctx->kv_dim, c.dtype, s);
      attention(ctx, ws.qkv, cache_l, ws.att, n_win, pos, 1, 1, s, true);
    }
    gemm(ctx, ws.att, L.wo, ws.x, rows, d, qd, kAddResidual, s);
    {
      ProfScope ps(ctx, kNorm, 0, s);
      launch_rmsnorm(ws.x, rows, d, c.rms_eps, ws.n, c.dtype, s);
    }
    if (ctx->fused_swiglu) {
      gemm(ctx, ws.n, L.wgu, ws.act, rows, 2 * (int64_t)F, d, kSwiGLU, s);
    } else {
      gemm(ctx, ws.n, L.wgu, ws.gu, rows, 2 * (int64_t)F, d, kStore, s);
      ProfScope ps(ctx, kNorm, 0, s);
      launch_swiglu(ws.gu, rows, F, ws.act, c.dtype, s);
    }
    gemm(ctx, ws.act, L.wdown, ws.x, rows, d, F, kAddResidual, s);
  }
  {
    ProfScope ps(ctx, kNorm, 0, s);
    launch_rmsnorm(ws.x, rows, d, c.rms_eps, ws.n, c.dtype, s);
  }
  gemm(ctx, ws.n, w_head, ctx->logits, rows, n_head, d, kStoreF32, s);
  ctx->row_max_valid = false;
}

// x = E[tok_in] for `rows` rows (and, on the fused-RMSNorm path, fp16(x) and its sums of squares)
static void embed_rows(lmgc_ctx* ctx, int64_t rows, cudaStream_t s) {
  const lmgc_config& c = ctx->cfg;
  if (ctx->fused_norm)
    launch_embed_fused(ctx->ws.tok_in, rows, ctx->w_embed, c.d_model, ctx->ws.x, (__half*)ctx->ws.n, ctx->ws.ss, s);
  else
    launch_embed(ctx->ws.tok_in, rows, ctx->w_embed, c.d_model, c.dtype, ctx->ws.x, s);
}

// Model logits for windows [first_win, first_win + nb) of a token stream, into ctx->logits.
static void forward_windows(lmgc_ctx* ctx, const uint16_t* tok, int64_t n_tok, int64_t first_win, int64_t nb,
                            cudaStream_t s, bool narrow = false) {
  const lmgc_config& c = ctx->cfg;
  const int64_t rows = nb * c.window;
  {
    ProfScope ps(ctx, kOther, 0, s);
    launch_window_inputs(tok, n_tok, first_win, nb, c.window, ctx->ws.tok_in, s);
    embed_rows(ctx, rows, s);
  }
  forward_layers(ctx, rows, nb, false, 0, s, narrow);
}

template <typename T>
static cudaError_t dmalloc(T** p, size_t bytes) {
  return cudaMalloc((void**)p, bytes ? bytes : 16);
}

template <typename T>
static cudaError_t ensure(T** p, size_t* cap, size_t need) {
  if (*cap >= need && *p) return cudaSuccess;
  if (*p) cudaFree(*p);
  *p = nullptr;
  *cap = 0;
  cudaError_t e = cudaMalloc((void**)p, need ? need : 16);
  if (e == cudaSuccess) *cap = need;
  return e;
}

static lmgc_status check_err_word(lmgc_ctx* ctx, cudaStream_t s, const char* what) {
  uint32_t h = 0;
  LMGC_CUDA(ctx, cudaMemcpyAsync(&h, ctx->d_err, 4, cudaMemcpyDeviceToHost, s));
  LMGC_CUDA(ctx, cudaStreamSynchronize(s));
  if (h == 0) return LMGC_OK;
  cudaMemsetAsync(ctx->d_err, 0, 4, s);
  cudaStreamSynchronize(s);
  if (h & kErrLimit) return fail(ctx, LMGC_ERR_LIMIT, std::string(what) + ": device loop limit");
  return fail(ctx, LMGC_ERR_CORRUPT, std::string(what) + ": corrupt input (device error word " +
                                         std::to_string(h) + ")");
}

__global__ void k_fill_win_len(uint32_t* wl, int64_t n_win, int64_t W, int64_t n_tok) {
  int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w < n_win) wl[w] = (uint32_t)(n_tok - w * W < W ? n_tok - w * W : W);
}

__global__ void k_dec_inputs(const uint16_t* __restrict__ dec_tok, int64_t n, int64_t W, int64_t pos,
                             uint16_t* __restrict__ tok_in) {
  int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w < n) tok_in[w] = pos == 0 ? (uint16_t)kTokBos : dec_tok[w * W + pos - 1];
}

}  // namespace lmgc

using namespace lmgc;

// ------------------------------------------------------------------------------------------
extern "C" {

lmgc_status lmgc_last_error(const lmgc_ctx* ctx, char* buf, size_t len) {
  if (!buf || !len) return LMGC_ERR_INVALID;
  const std::string& m = ctx ? ctx->err : g_thread_err;
  size_t n = std::min(len - 1, m.size());
  memcpy(buf, m.data(), n);
  buf[n] = 0;
  return LMGC_OK;
}

lmgc_status lmgc_tokens_per_value(const lmgc_ctx* ctx, size_t* tpv) {
  if (!ctx || !tpv) return LMGC_ERR_INVALID;
  const lmgc_config& c = ctx->cfg;
  const int64_t t1 = serial_tokens(c.input_kind, c.sep_mode, c.byte_group, 1);
  if (serial_tokens(c.input_kind, c.sep_mode, c.byte_group, 8) != 8 * t1)
    return fail(const_cast<lmgc_ctx*>(ctx), LMGC_ERR_INVALID, "byte groups cross values: no tokens-per-value count");
  *tpv = (size_t)t1;
  return LMGC_OK;
}

lmgc_status lmgc_serial_tokens(const lmgc_ctx* ctx, size_t n, size_t* n_tok) {
  if (!ctx || !n_tok) return LMGC_ERR_INVALID;
  *n_tok = (size_t)serial_tokens(ctx->cfg.input_kind, ctx->cfg.sep_mode, ctx->cfg.byte_group, (int64_t)n);
  return LMGC_OK;
}

lmgc_status lmgc_destroy(lmgc_ctx* ctx) {
  if (!ctx) return LMGC_OK;
  cudaDeviceSynchronize();
  void* ptrs[] = {ctx->weights_blob, ctx->rope_cs, ctx->exp2_tab, ctx->ws.x, ctx->ws.n, ctx->ws.qkv, ctx->ws.att,
                  ctx->ws.act, ctx->ws.gu, ctx->ws.ss, ctx->ws.tok_in, ctx->logits, ctx->row_max, ctx->d_err, ctx->tok, ctx->pair_start,
                  ctx->win_len, ctx->host_in, ctx->host_out, ctx->kv_cache, ctx->w_head_alpha};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  for (auto& e : ctx->ev)
    if (e) cudaEventDestroy(e);
  for (auto e : ctx->batch_ev) cudaEventDestroy(e);
  for (auto& r : ctx->prof.pending) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : ctx->prof.pool) cudaEventDestroy(e);
  delete ctx;
  return LMGC_OK;
}

lmgc_status lmgc_create(const lmgc_config* cfg, lmgc_ctx** out) {
  if (!cfg || !out) return fail(nullptr, LMGC_ERR_INVALID, "null argument");
  *out = nullptr;
  const lmgc_config& c = *cfg;
  if (c.n_layers < 0 || c.d_model <= 0 || c.n_heads <= 0 || c.n_kv_heads <= 0 || c.d_ffn <= 0 ||
      c.d_model % c.n_heads || c.n_heads % c.n_kv_heads || c.vocab < 20 || c.window < 1 || c.batch_windows < 1)
    return fail(nullptr, LMGC_ERR_INVALID, "bad model shape");
  const int hd = c.d_model / c.n_heads;
  if (c.dtype == LMGC_BF16 && hd != 64 && hd != 128)
    return fail(nullptr, LMGC_ERR_INVALID, "head dim of a bf16 model must be 64 or 128 (tcgen05 attention)");
  if (c.dtype != LMGC_BF16 && hd != 32 && hd != 64)
    return fail(nullptr, LMGC_ERR_INVALID, "head dim of an fp32 model must be 32 or 64 (tcgen05 TF32 attention)");
  if (c.d_model % 8 || c.d_ffn % 8) return fail(nullptr, LMGC_ERR_INVALID, "d_model and d_ffn must be multiples of 8");
  if (c.cdf_bits < 1 || c.cdf_bits > 30 || (int64_t)c.vocab >= (1ll << c.cdf_bits))
    return fail(nullptr, LMGC_ERR_INVALID, "cdf_bits must satisfy vocab < 2^cdf_bits <= 2^30");
  if (c.dtype != LMGC_F32 && c.dtype != LMGC_BF16) return fail(nullptr, LMGC_ERR_INVALID, "bad dtype");
  int tpv = tokens_per_value(c.input_kind, c.sep_mode);
  if (tpv < 0) return fail(nullptr, LMGC_ERR_INVALID, "bad input kind or separator mode");
  if (c.byte_group < 0 || c.byte_group > 8 || c.byte_order < 0 || c.byte_order > 1)
    return fail(nullptr, LMGC_ERR_INVALID, "byte_group must be 0..8 and byte_order 0 or 1");
  if (c.alphabet != 0 && c.alphabet != 1) return fail(nullptr, LMGC_ERR_INVALID, "alphabet must be 0 or 1");

  lmgc_ctx* ctx = new lmgc_ctx();
  ctx->cfg = c;
  if (c.alphabet) {
    // the 16 hex digits, then the separator ids of sep_mode in ascending order
    AlphaIds& a = ctx->alpha;
    for (a.n = 0; a.n < 16; a.n++) a.id[a.n] = a.n;
    if (c.sep_mode == LMGC_SEP_SPACE || c.sep_mode == LMGC_SEP_COMMA_SPACE) a.id[a.n++] = kTokSpace;
    if (c.sep_mode == LMGC_SEP_COMMA || c.sep_mode == LMGC_SEP_COMMA_SPACE) a.id[a.n++] = kTokComma;
    if (c.sep_mode == LMGC_SEP_SEMI) a.id[a.n++] = kTokSemi;
  }
  cudaGetDevice(&ctx->device);
  ctx->hd = hd;
  ctx->qkv_dim = (c.n_heads + 2 * c.n_kv_heads) * hd;
  ctx->kv_dim = 2 * c.n_kv_heads * hd;
  ctx->tpv = tpv;
  ctx->elt = c.dtype == LMGC_BF16 ? 2 : 4;
  if (c.dtype == LMGC_BF16) {
    // a bf16 model has one backend, the tcgen05 kernels: without the tensor-map encoder (or on a
    // device they do not run on) the context is refused instead of computing another way
    const bool tc = tc_attention_supported(hd, ctx->qkv_dim) && tc_attention_supported(hd, ctx->kv_dim) &&
                    tc_gemm_supported(1, ctx->qkv_dim, c.d_model, kStore) &&
                    tc_gemm_supported(1, c.d_model, (int64_t)c.n_heads * hd, kAddResidual) &&
                    tc_gemm_supported(1, 2 * (int64_t)c.d_ffn, c.d_model, kStore) &&
                    tc_gemm_supported(1, c.d_model, c.d_ffn, kAddResidual) &&
                    tc_gemm_supported(1, c.vocab, c.d_model, kStoreF32);
    if (!tc) {
      delete ctx;
      return fail(nullptr, LMGC_ERR_INVALID,
                  "bf16 models need the tcgen05 kernels: a Blackwell device and the driver's tensor-map encoder");
    }
  } else {
    // an fp32 model's contractions run on the tcgen05 TF32 kernel, likewise with no other backend
    const bool tc = tf32_attention_supported(hd, ctx->qkv_dim, ctx->qkv_dim) &&
                    tf32_attention_supported(hd, ctx->qkv_dim, ctx->kv_dim) &&
                    tf32_gemm_supported(1, ctx->qkv_dim, c.d_model) &&
                    tf32_gemm_supported(1, c.d_model, (int64_t)c.n_heads * hd) &&
                    tf32_gemm_supported(1, 2 * (int64_t)c.d_ffn, c.d_model) &&
                    tf32_gemm_supported(1, c.d_model, c.d_ffn) && tf32_gemm_supported(1, c.vocab, c.d_model);
    if (!tc) {
      delete ctx;
      return fail(nullptr, LMGC_ERR_INVALID,
                  "fp32 models need the tcgen05 TF32 kernels: a Blackwell device, the driver's tensor-map encoder "
                  "and inner dimensions that are multiples of 4");
    }
  }
  ctx->fused_rope = c.dtype == LMGC_BF16 && tc_gemm_supported(1, ctx->qkv_dim, c.d_model, kQKVRope);
  ctx->fused_norm = c.dtype == LMGC_BF16 && c.d_model % 256 == 0;
  ctx->fused_swiglu = c.dtype == LMGC_BF16 && c.d_ffn % 128 == 0 && tc_gemm_supported(1, 2 * c.d_ffn, c.d_model, kSwiGLU);
  const int64_t d = c.d_model, F = c.d_ffn, V = c.vocab, qd = (int64_t)c.n_heads * hd;
  const size_t e = ctx->elt;
  // weights: one blob, every tensor 256-byte aligned
  auto al = [](size_t x) { return (x + 255) / 256 * 256; };
  size_t off = 0;
  std::vector<size_t> offs;
  offs.push_back(off); off += al(V * d * e);                        // embed
  for (int l = 0; l < c.n_layers; l++) {
    offs.push_back(off); off += al((size_t)ctx->qkv_dim * d * e);   // wqkv
    offs.push_back(off); off += al((size_t)d * qd * e);             // wo
    offs.push_back(off); off += al((size_t)2 * F * d * e);          // wgu
    offs.push_back(off); off += al((size_t)d * F * e);              // wdown
  }
  offs.push_back(off); off += al(V * d * e);                        // head
  cudaStream_t s = 0;
  cudaError_t err = cudaMalloc(&ctx->weights_blob, off);
  if (err != cudaSuccess) {
    lmgc_destroy(ctx);
    return cuda_fail(nullptr, err, "weights");
  }
  char* base = (char*)ctx->weights_blob;
  int k = 0;
  ctx->w_embed = base + offs[k++];
  ctx->layers.resize(c.n_layers);
  for (int l = 0; l < c.n_layers; l++) {
    ctx->layers[l].wqkv = base + offs[k++];
    ctx->layers[l].wo = base + offs[k++];
    ctx->layers[l].wgu = base + offs[k++];
    ctx->layers[l].wdown = base + offs[k++];
  }
  ctx->w_head = base + offs[k++];
  // tensor ids: 0 embed, 1+7l+{q,k,v,o,gate,up,down}, 1+7L head; index = row-major canonical
  const uint64_t seed = c.weight_seed;
  const int dt = c.dtype;
  launch_init_weights(ctx->w_embed, dt, seed, 0, V, d, d, 0, c.init_std, s);
  for (int l = 0; l < c.n_layers; l++) {
    const uint32_t t = 1 + 7 * l;
    const Layer& L = ctx->layers[l];
    launch_init_weights(L.wqkv, dt, seed, t + 0, qd, d, d, 0, c.init_std, s);
    launch_init_weights(L.wqkv, dt, seed, t + 1, (int64_t)c.n_kv_heads * hd, d, d, qd, c.init_std, s);
    launch_init_weights(L.wqkv, dt, seed, t + 2, (int64_t)c.n_kv_heads * hd, d, d,
                        qd + (int64_t)c.n_kv_heads * hd, c.init_std, s);
    launch_init_weights(L.wo, dt, seed, t + 3, d, qd, qd, 0, c.init_std, s);
    if (ctx->fused_swiglu) {  // gate/up interleaved in 128-row blocks
      launch_init_weights(L.wgu, dt, seed, t + 4, F, d, d, 0, c.init_std, s, 128, 256);
      launch_init_weights(L.wgu, dt, seed, t + 5, F, d, d, 128, c.init_std, s, 128, 256);
    } else {
      launch_init_weights(L.wgu, dt, seed, t + 4, F, d, d, 0, c.init_std, s);
      launch_init_weights(L.wgu, dt, seed, t + 5, F, d, d, F, c.init_std, s);
    }
    launch_init_weights(L.wdown, dt, seed, t + 6, d, F, F, 0, c.init_std, s);
  }
  launch_init_weights(ctx->w_head, dt, seed, 1 + 7 * c.n_layers, V, d, d, 0, c.init_std, s);
  if (c.alphabet) {
    // the restricted alphabet's rows of the vocabulary weight in their order, zero rows after
    const size_t row = (size_t)d * ctx->elt;
    err = cudaMalloc(&ctx->w_head_alpha, kAlphaCols * row);
    if (err == cudaSuccess) err = cudaMemsetAsync(ctx->w_head_alpha, 0, kAlphaCols * row, s);
    for (int j = 0; j < ctx->alpha.n && err == cudaSuccess; j++)
      err = cudaMemcpyAsync((char*)ctx->w_head_alpha + j * row, (const char*)ctx->w_head + ctx->alpha.id[j] * row, row,
                            cudaMemcpyDeviceToDevice, s);
    ctx->alpha_cols.n = ctx->alpha.n;
    for (int j = 0; j < ctx->alpha.n; j++) ctx->alpha_cols.id[j] = j;
  }
  // RoPE table: angle pos * theta^(-2i/hd) in binary64, stored as fp32 (cos, sin)
  {
    std::vector<float2> cs((size_t)c.window * (hd / 2));
    for (int64_t p = 0; p < c.window; p++)
      for (int i = 0; i < hd / 2; i++) {
        double ang = (double)p * pow((double)c.rope_theta, -2.0 * i / hd);
        cs[p * (hd / 2) + i] = make_float2((float)cos(ang), (float)sin(ang));
      }
    err = cudaMalloc(&ctx->rope_cs, cs.size() * sizeof(float2));
    if (err == cudaSuccess) err = cudaMemcpy(ctx->rope_cs, cs.data(), cs.size() * sizeof(float2), cudaMemcpyHostToDevice);
  }
  if (err == cudaSuccess) err = cudaMalloc(&ctx->exp2_tab, 512 * sizeof(uint32_t));
  if (err == cudaSuccess) upload_exp2_tables(ctx->exp2_tab, s);
  if (err == cudaSuccess) err = cudaMalloc(&ctx->d_err, 16);
  if (err == cudaSuccess) err = cudaMemset(ctx->d_err, 0, 16);
  // workspace for batch_windows windows
  Workspace& ws = ctx->ws;
  ws.rows = (int64_t)c.batch_windows * c.window;
  const size_t R = (size_t)ws.rows;
  if (err == cudaSuccess) err = dmalloc(&ws.x, R * d * 4);
  if (err == cudaSuccess) err = dmalloc(&ws.n, R * d * e);
  if (err == cudaSuccess) err = dmalloc(&ws.qkv, R * ctx->qkv_dim * e);
  if (err == cudaSuccess) err = dmalloc(&ws.att, R * qd * e);
  if (err == cudaSuccess) err = dmalloc(&ws.act, R * F * e);
  if (err == cudaSuccess && !ctx->fused_swiglu) err = dmalloc(&ws.gu, R * 2 * F * e);
  ctx->fused_norm = ctx->fused_norm && ctx->fused_rope && ctx->fused_swiglu;
  if (err == cudaSuccess && ctx->fused_norm) err = dmalloc(&ws.ss, R * (size_t)(d / 128) * 4);
  if (err == cudaSuccess) err = dmalloc(&ws.tok_in, R * 2);
  // [R][V], or [R][kAlphaCols] rows of the narrow head when that is wider
  if (err == cudaSuccess) err = dmalloc(&ctx->logits, R * std::max<int64_t>(V, kAlphaCols) * 4);
  if (err == cudaSuccess) err = dmalloc(&ctx->row_max, R * 4);
  for (int i = 0; i < 6 && err == cudaSuccess; i++) err = cudaEventCreate(&ctx->ev[i]);
  if (err == cudaSuccess) err = cudaDeviceSynchronize();
  if (err == cudaSuccess) err = cudaGetLastError();
  if (err != cudaSuccess) {
    lmgc_destroy(ctx);
    return cuda_fail(nullptr, err, "lmgc_create");
  }
  for (int i = 0; i < kNumClasses; i++) ctx->prof.stats[i] = KernelStat{kClassNames[i], 0, 0.f, 0.0};
  *out = ctx;
  return LMGC_OK;
}

lmgc_status lmgc_serialize(lmgc_ctx* ctx, const void* d_in, size_t n, uint16_t* d_tok, size_t cap_tok,
                           size_t* n_tok, lmgc_stream stream) {
  if (!ctx || !n_tok || (n && (!d_in || !d_tok))) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  const lmgc_config& c = ctx->cfg;
  size_t need = (size_t)serial_tokens(c.input_kind, c.sep_mode, c.byte_group, (int64_t)n);
  *n_tok = need;
  if (cap_tok < need) return fail(ctx, LMGC_ERR_NO_SPACE, "token buffer too small");
  cudaStream_t s = (cudaStream_t)stream;
  launch_serialize(c.input_kind, c.sep_mode, c.byte_group, c.byte_order, d_in, (int64_t)n, d_tok, s);
  LMGC_CUDA(ctx, cudaGetLastError());
  return LMGC_OK;
}

lmgc_status lmgc_deserialize(lmgc_ctx* ctx, const uint16_t* d_tok, size_t n_tok, void* d_out, size_t cap_values,
                             size_t* n_values, lmgc_stream stream) {
  if (!ctx || !n_values || (n_tok && (!d_tok || !d_out))) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  const lmgc_config& c = ctx->cfg;
  const int64_t nvs = serial_values(c.input_kind, c.sep_mode, c.byte_group, (int64_t)n_tok);
  if (nvs < 0) return fail(ctx, LMGC_ERR_CORRUPT, "no value count serialises to this many tokens");
  size_t nv = (size_t)nvs;
  *n_values = nv;
  if (cap_values < nv) return fail(ctx, LMGC_ERR_NO_SPACE, "value buffer too small");
  cudaStream_t s = (cudaStream_t)stream;
  launch_deserialize(c.input_kind, c.sep_mode, c.byte_group, c.byte_order, d_tok, (int64_t)nv, d_out, ctx->d_err, s);
  LMGC_CUDA(ctx, cudaGetLastError());
  return check_err_word(ctx, s, "deserialize");
}

lmgc_status lmgc_lm_probs(lmgc_ctx* ctx, const uint16_t* d_tok, size_t n_tok, size_t first_win, size_t n_win,
                          float* d_logits, lmgc_stream stream) {
  if (!ctx || !d_tok || !d_logits) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  const int64_t W = ctx->cfg.window, V = ctx->cfg.vocab;
  const int64_t total_win = ((int64_t)n_tok + W - 1) / W;
  if ((int64_t)(first_win + n_win) > total_win) return fail(ctx, LMGC_ERR_INVALID, "window range beyond the stream");
  cudaStream_t s = (cudaStream_t)stream;
  for (int64_t w0 = 0; w0 < (int64_t)n_win; w0 += ctx->cfg.batch_windows) {
    int64_t nb = std::min<int64_t>(ctx->cfg.batch_windows, (int64_t)n_win - w0);
    forward_windows(ctx, d_tok, (int64_t)n_tok, (int64_t)first_win + w0, nb, s);
    LMGC_CUDA(ctx, cudaMemcpyAsync(d_logits + w0 * W * V, ctx->logits, (size_t)(nb * W * V) * 4,
                                   cudaMemcpyDeviceToDevice, s));
  }
  LMGC_CUDA(ctx, cudaGetLastError());
  if (ctx->prof.enabled) {
    cudaStreamSynchronize(s);
    prof_collect(ctx);
  }
  return LMGC_OK;
}

lmgc_status lmgc_quantize_cdf(lmgc_ctx* ctx, const float* d_logits, size_t rows, uint32_t* d_cdf,
                              lmgc_stream stream) {
  if (!ctx || (rows && (!d_logits || !d_cdf))) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  launch_quantize_cdf(d_logits, (int64_t)rows, ctx->cfg.vocab, ctx->cfg.cdf_bits, ctx->exp2_tab, d_cdf,
                      (cudaStream_t)stream);
  LMGC_CUDA(ctx, cudaGetLastError());
  return LMGC_OK;
}

lmgc_status lmgc_cdf_pairs(lmgc_ctx* ctx, const float* d_logits, size_t rows, const uint16_t* d_sym,
                           uint32_t* d_start, uint32_t* d_freq, lmgc_stream stream) {
  if (!ctx || (rows && (!d_logits || !d_sym || !d_start || !d_freq)))
    return fail(ctx, LMGC_ERR_INVALID, "null argument");
  if (ctx->cfg.alphabet) {
    launch_cdf_pairs_alpha(d_logits, (int64_t)rows, ctx->cfg.vocab, ctx->cfg.cdf_bits, ctx->exp2_tab, d_sym, 0, 1, 0,
                           d_start, d_freq, 0, (cudaStream_t)stream, 0, ctx->alpha, ctx->d_err);
    LMGC_CUDA(ctx, cudaGetLastError());
    return check_err_word(ctx, (cudaStream_t)stream, "cdf_pairs");
  }
  // the encode's kernel, with each row's maximum from a pass of its own (stream-ordered scratch)
  cudaStream_t s = (cudaStream_t)stream;
  if (rows == 0) return LMGC_OK;
  uint32_t* keys = nullptr;
  LMGC_CUDA(ctx, cudaMallocAsync((void**)&keys, rows * 4, s));
  launch_cdf_pairs(d_logits, (int64_t)rows, ctx->cfg.vocab, ctx->cfg.cdf_bits, ctx->exp2_tab, d_sym, 0, 1, 0,
                   d_start, d_freq, 0, s, 0, keys, false);
  const cudaError_t e = cudaGetLastError();
  cudaFreeAsync(keys, s);
  LMGC_CUDA(ctx, e);
  return LMGC_OK;
}

}  // extern "C"

// lmgc_range_encode and lmgc_range_encode_tiled: the coder over a caller's pairs (validated
// unless the caller vouches for them), with stream-ordered scratch
static lmgc_status range_encode_any(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                                    size_t win_tokens, const uint32_t* d_win_len, size_t stride_win,
                                    size_t stride_pos, bool tiled, bool validate, uint8_t* d_out, size_t cap,
                                    size_t* out_bytes, uint32_t* d_bitlen, lmgc_stream stream) {
  if (!out_bytes || (n_win && (!d_start || !d_freq || !d_bitlen)))
    return fail(nullptr, LMGC_ERR_INVALID, "null argument");
  if (cdf_bits < 1 || cdf_bits > 30) return fail(nullptr, LMGC_ERR_INVALID, "cdf_bits must be in 1..30");
  *out_bytes = 0;
  if (n_win == 0) return LMGC_OK;
  // the tiles are staged by bulk copies, whose sources must be 16-byte aligned
  if (tiled && (((uintptr_t)d_start | (uintptr_t)d_freq) & 15))
    return fail(nullptr, LMGC_ERR_INVALID, "range_encode_tiled: pair arrays must be 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  const size_t slot = slot_bytes(win_tokens, cdf_bits);
  uint8_t* slots = nullptr;
  uint64_t* offs = nullptr;
  uint32_t* derr = nullptr;
  // the tiled coder keeps each 32-window block's slots as one interleaved table: whole blocks
  cudaError_t e = cudaMallocAsync((void**)&slots, slot * (tiled ? (n_win + 31) / 32 * 32 : n_win), s);
  if (e == cudaSuccess) e = cudaMallocAsync((void**)&offs, (n_win + 1) * 8 + 16, s);
  if (e == cudaSuccess) e = cudaMallocAsync((void**)&derr, 16, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(derr, 0, 4, s);
  lmgc_status st = LMGC_OK;
  if (e != cudaSuccess) {
    st = cuda_fail(nullptr, e, "range_encode scratch");
  } else {
    {
      ProfScope ps(nullptr, kCoder, 8.0 * (double)n_win * (double)win_tokens, s);
      launch_range_encode(d_start, d_freq, cdf_bits, (int64_t)n_win, (int64_t)win_tokens, d_win_len,
                          (int64_t)stride_win, (int64_t)stride_pos, slots, slot, d_bitlen, derr, s, tiled,
                          validate);
    }
    launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, nullptr, s, tiled);
    uint64_t total = 0;
    uint32_t herr = 0;
    e = cudaMemcpyAsync(&total, offs + n_win, 8, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, derr, 4, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) st = cuda_fail(nullptr, e, "range_encode");
    else if (herr) st = fail(nullptr, LMGC_ERR_INVALID, "range_encode: invalid (start, freq) or window length");
    else {
      *out_bytes = total;
      if (cap < total) st = fail(nullptr, LMGC_ERR_NO_SPACE, "range_encode: output too small");
      else {
        launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, d_out, s, tiled);
        e = cudaGetLastError();
        if (e != cudaSuccess) st = cuda_fail(nullptr, e, "range_encode pack");
      }
    }
  }
  if (slots) cudaFreeAsync(slots, s);
  if (offs) cudaFreeAsync(offs, s);
  if (derr) cudaFreeAsync(derr, s);
  cudaStreamSynchronize(s);
  if (free_ctx()->prof.enabled) prof_collect(free_ctx());
  return st;
}

extern "C" {

lmgc_status lmgc_range_encode(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                              size_t win_tokens, const uint32_t* d_win_len, size_t stride_win, size_t stride_pos,
                              uint8_t* d_out, size_t cap, size_t* out_bytes, uint32_t* d_bitlen,
                              lmgc_stream stream) {
  return range_encode_any(d_start, d_freq, cdf_bits, n_win, win_tokens, d_win_len, stride_win, stride_pos, false,
                          true, d_out, cap, out_bytes, d_bitlen, stream);
}

lmgc_status lmgc_range_encode_tiled(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                                    size_t win_tokens, const uint32_t* d_win_len, int validate, uint8_t* d_out,
                                    size_t cap, size_t* out_bytes, uint32_t* d_bitlen, lmgc_stream stream) {
  return range_encode_any(d_start, d_freq, cdf_bits, n_win, win_tokens, d_win_len, 0, 0, true, validate != 0, d_out,
                          cap, out_bytes, d_bitlen, stream);
}

lmgc_status lmgc_pair_tile_elems(size_t n_win, size_t win_tokens, size_t* elems) {
  if (!elems) return LMGC_ERR_INVALID;
  *elems = (size_t)pair_tile_elems((int64_t)n_win, (int64_t)win_tokens);
  return LMGC_OK;
}

lmgc_status lmgc_encode_bound(const lmgc_ctx* ctx, size_t n, size_t* bytes) {
  if (!ctx || !bytes) return LMGC_ERR_INVALID;
  const size_t n_tok = (size_t)n_tokens(ctx, (int64_t)n), W = (size_t)ctx->cfg.window;
  const size_t n_win = (n_tok + W - 1) / W;
  *bytes = 64 + 8 * n_win + (n_tok * (size_t)ctx->cfg.cdf_bits + 2 * n_win + 7) / 8 + n_win;
  return LMGC_OK;
}

}  // extern "C"

namespace lmgc {

// Phase 1 of an encode: serialise all n values, then model, CDF pairs and coder for the windows
// [w_begin, w_begin + w_count) of the token stream. The codes stay in the context's slot scratch;
// *payload receives their packed size. Phase 2 (encode_pack) writes them out.
static lmgc_status encode_codes(lmgc_ctx* ctx, const void* d_in, size_t n, int64_t w_begin, int64_t w_count,
                                uint64_t* payload, cudaStream_t s) {
  const lmgc_config& c = ctx->cfg;
  const int64_t W = c.window, P = c.cdf_bits;
  const int64_t n_tok = n_tokens(ctx, (int64_t)n);
  const int64_t n_win = w_count;
  const size_t slot = slot_bytes((size_t)W, (int)P);
  // staging (grown on demand; reused across calls)
  LMGC_CUDA(ctx, ensure(&ctx->tok, &ctx->tok_cap, (size_t)n_tok * 2 + 16));
  // (start, freq) pairs in the coder's window tiles (whole tiles: 32-window blocks, 8-position groups)
  const size_t pair_elems = (size_t)pair_tile_elems(n_win, W);
  LMGC_CUDA(ctx, ensure(&ctx->pair_start, &ctx->pair_cap, 2 * pair_elems * 4));
  ctx->pair_freq = ctx->pair_start + pair_elems;
  // win_len [n_win] u32 | bitlen [n_win] u32 | token crc [n_win] u32 | offsets [n_win+1] u64 | slots
  const size_t tbl = ((size_t)n_win * 4 + 255) / 256 * 256;
  const size_t wl_off = 0, bl_off = tbl, cr_off = 2 * tbl, of_off = 3 * tbl,
               sl_off = of_off + (((size_t)n_win + 1) * 8 + 255) / 256 * 256;
  // the tiled coder keeps each 32-window block's slots as one interleaved table: whole blocks
  LMGC_CUDA(ctx, ensure(&ctx->win_len, &ctx->win_cap, sl_off + slot * (((size_t)n_win + 31) / 32 * 32)));
  uint32_t* d_wl = (uint32_t*)((char*)ctx->win_len + wl_off);
  ctx->enc_bl = (uint32_t*)((char*)ctx->win_len + bl_off);
  ctx->enc_crc = (uint32_t*)((char*)ctx->win_len + cr_off);
  ctx->enc_off = (uint64_t*)((char*)ctx->win_len + of_off);
  ctx->enc_slots = (uint8_t*)ctx->win_len + sl_off;
  ctx->enc_slot = slot;
  ctx->enc_nwin = n_win;

  LMGC_CUDA(ctx, cudaEventRecord(ctx->ev[0], s));
  {
    ProfScope ps(ctx, kSer, (double)n * (ctx->cfg.input_kind == LMGC_IN_F32 ? 4 : 1) + (double)n_tok * 2, s);
    launch_serialize(c.input_kind, c.sep_mode, c.byte_group, c.byte_order, d_in, (int64_t)n, ctx->tok, s);
  }
  LMGC_CUDA(ctx, cudaEventRecord(ctx->ev[1], s));
  const int64_t n_batches = (n_win + c.batch_windows - 1) / c.batch_windows;
  while ((int64_t)ctx->batch_ev.size() < 2 * n_batches + 1) {
    cudaEvent_t e;
    LMGC_CUDA(ctx, cudaEventCreate(&e));
    ctx->batch_ev.push_back(e);
  }
  cudaEventRecord(ctx->batch_ev[0], s);
  for (int64_t b = 0; b < n_batches; b++) {
    const int64_t w0 = w_begin + b * c.batch_windows;
    const int64_t nb = std::min<int64_t>(c.batch_windows, w_begin + n_win - w0);
    forward_windows(ctx, ctx->tok, n_tok, w0, nb, s, c.alphabet != 0);
    cudaEventRecord(ctx->batch_ev[2 * b + 1], s);
    {
      const int64_t rows = nb * W;
      // per row: the logits the quantiser reads (the alphabet's ids only with alphabet 1), the
      // token and the pair
      const double cols = c.alphabet ? (double)ctx->alpha.n : (double)c.vocab;
      ProfScope ps(ctx, kCdf, (double)rows * (cols * 4 + 2 + 8), s);
      if (c.alphabet)
        launch_cdf_pairs_alpha(ctx->logits, rows, kAlphaCols, (int)P, ctx->exp2_tab, ctx->tok, n_tok, (int)W, w0,
                               ctx->pair_start, ctx->pair_freq, 1, s, w_begin, ctx->alpha_cols, ctx->d_err);
      else
        launch_cdf_pairs(ctx->logits, rows, c.vocab, (int)P, ctx->exp2_tab, ctx->tok, n_tok, (int)W, w0,
                         ctx->pair_start, ctx->pair_freq, 1, s, w_begin, ctx->row_max, ctx->row_max_valid);
    }
    cudaEventRecord(ctx->batch_ev[2 * b + 2], s);
  }
  LMGC_CUDA(ctx, cudaEventRecord(ctx->ev[2], s));
  note_launch();
  k_fill_win_len<<<(unsigned)((n_win + 255) / 256), 256, 0, s>>>(d_wl, n_win, W, n_tok - w_begin * W);
  launch_window_crc(ctx->tok + w_begin * W, W, d_wl, n_win, ctx->enc_crc, s);
  {
    ProfScope ps(ctx, kCoder, (double)n_win * (double)W * 8, s);
    // the pairs come from the CDF kernels, valid by construction: no per-pair check
    launch_range_encode(ctx->pair_start, ctx->pair_freq, (int)P, n_win, W, d_wl, 0, 0, ctx->enc_slots, slot,
                        ctx->enc_bl, ctx->d_err, s, true, false);
  }
  LMGC_CUDA(ctx, cudaEventRecord(ctx->ev[3], s));
  launch_pack_codes(ctx->enc_slots, slot, ctx->enc_bl, n_win, ctx->enc_off, nullptr, s, true);
  LMGC_CUDA(ctx, cudaMemcpyAsync(payload, ctx->enc_off + n_win, 8, cudaMemcpyDeviceToHost, s));
  lmgc_status st = check_err_word(ctx, s, "encode");
  ctx->enc_batches = n_batches;
  return st;
}

// Phase 2: the codes of the last encode_codes call, byte-aligned in window order, to d_payload;
// their bit lengths to d_bitlen and their token checksums to d_crc (device).
static lmgc_status encode_pack(lmgc_ctx* ctx, uint8_t* d_payload, uint32_t* d_bitlen, uint32_t* d_crc,
                               cudaStream_t s) {
  const int64_t n_win = ctx->enc_nwin;
  LMGC_CUDA(ctx, cudaMemcpyAsync(d_bitlen, ctx->enc_bl, 4 * (size_t)n_win, cudaMemcpyDeviceToDevice, s));
  LMGC_CUDA(ctx, cudaMemcpyAsync(d_crc, ctx->enc_crc, 4 * (size_t)n_win, cudaMemcpyDeviceToDevice, s));
  launch_pack_codes(ctx->enc_slots, ctx->enc_slot, ctx->enc_bl, n_win, ctx->enc_off, d_payload, s, true);
  LMGC_CUDA(ctx, cudaEventRecord(ctx->ev[5], s));
  LMGC_CUDA(ctx, cudaStreamSynchronize(s));
  LMGC_CUDA(ctx, cudaGetLastError());
  float x = 0.f, ms_lm = 0.f, ms_cdf = 0.f;
  for (int64_t b = 0; b < ctx->enc_batches; b++) {
    cudaEventElapsedTime(&x, ctx->batch_ev[2 * b], ctx->batch_ev[2 * b + 1]);
    ms_lm += x;
    cudaEventElapsedTime(&x, ctx->batch_ev[2 * b + 1], ctx->batch_ev[2 * b + 2]);
    ms_cdf += x;
  }
  cudaEventElapsedTime(&x, ctx->ev[0], ctx->ev[1]);
  ctx->stage_ms[0] = x;
  ctx->stage_ms[1] = ms_lm;
  ctx->stage_ms[2] = ms_cdf;
  cudaEventElapsedTime(&x, ctx->ev[2], ctx->ev[3]);
  ctx->stage_ms[3] = x;
  cudaEventElapsedTime(&x, ctx->ev[3], ctx->ev[5]);
  ctx->stage_ms[4] = x;
  if (ctx->prof.enabled) prof_collect(ctx);
  return LMGC_OK;
}

constexpr uint32_t kContainerVersion = 2;  // 2: per-window token checksums after the bit lengths

// header word at byte 36: the separator mode, and the byte grouping (0 for the default layout)
static uint32_t serial_word(const lmgc_config& c) {
  return (uint32_t)c.sep_mode | (uint32_t)c.byte_group << 8 | (uint32_t)c.byte_order << 16 |
         (uint32_t)c.alphabet << 24;
}

static void container_header(const lmgc_ctx* ctx, size_t n, uint8_t* h) {
  const lmgc_config& c = ctx->cfg;
  const uint64_t n_tok = (uint64_t)n_tokens(ctx, (int64_t)n);
  const uint64_t n_win = (n_tok + (uint64_t)c.window - 1) / (uint64_t)c.window;
  memset(h, 0, 64);
  uint32_t u32;
  uint64_t u64;
  memcpy(h, "LMGC", 4);
  u32 = kContainerVersion; memcpy(h + 4, &u32, 4);
  u64 = n; memcpy(h + 8, &u64, 8);
  u64 = n_tok; memcpy(h + 16, &u64, 8);
  u32 = (uint32_t)c.window; memcpy(h + 24, &u32, 4);
  u32 = (uint32_t)c.cdf_bits; memcpy(h + 28, &u32, 4);
  u32 = (uint32_t)c.input_kind; memcpy(h + 32, &u32, 4);
  u32 = serial_word(c); memcpy(h + 36, &u32, 4);
  u32 = (uint32_t)c.vocab; memcpy(h + 40, &u32, 4);
  u32 = (uint32_t)n_win; memcpy(h + 44, &u32, 4);
  u64 = c.weight_seed; memcpy(h + 48, &u64, 8);
  u32 = model_crc(c); memcpy(h + 56, &u32, 4);
  u32 = crc32(h, 60); memcpy(h + 60, &u32, 4);
}

}  // namespace lmgc

extern "C" {

lmgc_status lmgc_encode(lmgc_ctx* ctx, const void* d_in, size_t n, uint8_t* d_out, size_t cap, size_t* out_bytes,
                        lmgc_stream stream) {
  if (!ctx || !d_in || !out_bytes) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  if (n == 0) return fail(ctx, LMGC_ERR_INVALID, "empty input");
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t W = ctx->cfg.window;
  const int64_t n_win = (n_tokens(ctx, (int64_t)n) + W - 1) / W;
  uint64_t payload = 0;
  lmgc_status st = encode_codes(ctx, d_in, n, 0, n_win, &payload, s);
  if (st != LMGC_OK) return st;
  const size_t total = 64 + 8 * (size_t)n_win + payload;
  *out_bytes = total;
  if (cap < total || !d_out) return fail(ctx, LMGC_ERR_NO_SPACE, "container buffer too small");
  uint8_t h[64];
  container_header(ctx, n, h);
  LMGC_CUDA(ctx, cudaMemcpyAsync(d_out, h, 64, cudaMemcpyHostToDevice, s));
  return encode_pack(ctx, d_out + 64 + 8 * (size_t)n_win, (uint32_t*)(d_out + 64),
                     (uint32_t*)(d_out + 64 + 4 * (size_t)n_win), s);
}

lmgc_status lmgc_encode_windows(lmgc_ctx* ctx, const void* d_in, size_t n, size_t first_win, size_t n_win,
                                uint8_t* d_payload, size_t cap, size_t* payload_bytes, uint32_t* d_bitlen,
                                uint32_t* d_crc, lmgc_stream stream) {
  if (!ctx || !d_in || !payload_bytes || (n_win && (!d_bitlen || !d_crc)))
    return fail(ctx, LMGC_ERR_INVALID, "null argument");
  const int64_t W = ctx->cfg.window;
  const int64_t total_win = (n_tokens(ctx, (int64_t)n) + W - 1) / W;
  if (n == 0 || n_win == 0 || (int64_t)(first_win + n_win) > total_win)
    return fail(ctx, LMGC_ERR_INVALID, "window range outside the stream");
  cudaStream_t s = (cudaStream_t)stream;
  uint64_t payload = 0;
  lmgc_status st = encode_codes(ctx, d_in, n, (int64_t)first_win, (int64_t)n_win, &payload, s);
  if (st != LMGC_OK) return st;
  *payload_bytes = payload;
  if (cap < payload || !d_payload) return fail(ctx, LMGC_ERR_NO_SPACE, "payload buffer too small");
  return encode_pack(ctx, d_payload, d_bitlen, d_crc, s);
}

lmgc_status lmgc_container_header(const lmgc_ctx* ctx, size_t n, uint8_t* h_header) {
  if (!ctx || !h_header) return LMGC_ERR_INVALID;
  container_header(ctx, n, h_header);
  return LMGC_OK;
}

lmgc_status lmgc_encode_host(lmgc_ctx* ctx, const void* h_in, size_t n, uint8_t* h_out, size_t cap,
                             size_t* out_bytes, lmgc_stream stream) {
  if (!ctx || !h_in || !out_bytes) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  cudaStream_t s = (cudaStream_t)stream;
  const size_t in_bytes = n * (ctx->cfg.input_kind == LMGC_IN_F32 ? 4 : 1);
  size_t bound = 0;
  lmgc_encode_bound(ctx, n, &bound);
  LMGC_CUDA(ctx, ensure(&ctx->host_in, &ctx->host_in_cap, in_bytes));
  LMGC_CUDA(ctx, ensure(&ctx->host_out, &ctx->host_out_cap, bound));
  LMGC_CUDA(ctx, cudaMemcpyAsync(ctx->host_in, h_in, in_bytes, cudaMemcpyHostToDevice, s));
  lmgc_status st = lmgc_encode(ctx, ctx->host_in, n, ctx->host_out, ctx->host_out_cap, out_bytes, stream);
  if (st != LMGC_OK) return st;
  if (cap < *out_bytes || !h_out) return fail(ctx, LMGC_ERR_NO_SPACE, "host container buffer too small");
  LMGC_CUDA(ctx, cudaMemcpyAsync(h_out, ctx->host_out, *out_bytes, cudaMemcpyDeviceToHost, s));
  LMGC_CUDA(ctx, cudaStreamSynchronize(s));
  return LMGC_OK;
}

// bytes of KV cache one decoded window needs: every layer's keys and values at W positions
static size_t decode_kv_per_window(const lmgc_ctx* ctx) {
  return (size_t)std::max(1, ctx->cfg.n_layers) * (size_t)ctx->cfg.window * (size_t)ctx->kv_dim * ctx->elt;
}

// windows per decode batch: a KV cache of half the free device memory (or the context's cache if
// larger), at most one workspace row per window (batch_windows * W rows)
static cudaError_t decode_batch(const lmgc_ctx* ctx, size_t* n) {
  size_t free_b = 0, total_b = 0;
  const cudaError_t e = cudaMemGetInfo(&free_b, &total_b);
  if (e != cudaSuccess) return e;
  const size_t budget = std::max<size_t>(ctx->kv_cap, free_b / 2);
  *n = std::min<size_t>(budget / decode_kv_per_window(ctx), (size_t)ctx->cfg.batch_windows * ctx->cfg.window);
  return cudaSuccess;
}

lmgc_status lmgc_decode(lmgc_ctx* ctx, const uint8_t* d_in, size_t in_bytes, const uint32_t* h_win_ids,
                        size_t n_ids, uint16_t* d_tok, size_t cap_tok, lmgc_stream stream) {
  if (!ctx || !d_in || (n_ids && (!h_win_ids || !d_tok))) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  const lmgc_config& c = ctx->cfg;
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t W = c.window;
  if (in_bytes < 64) return fail(ctx, LMGC_ERR_CORRUPT, "container shorter than its header");
  uint8_t h[64];
  LMGC_CUDA(ctx, cudaMemcpyAsync(h, d_in, 64, cudaMemcpyDeviceToHost, s));
  LMGC_CUDA(ctx, cudaStreamSynchronize(s));
  uint32_t hcrc, mcrc, ver, hW, hP, kind, sep, vocab, n_win;
  uint64_t n_tok;
  memcpy(&hcrc, h + 60, 4);
  if (memcmp(h, "LMGC", 4) || hcrc != crc32(h, 60)) return fail(ctx, LMGC_ERR_CORRUPT, "bad container header");
  memcpy(&ver, h + 4, 4);
  memcpy(&n_tok, h + 16, 8);
  memcpy(&hW, h + 24, 4);
  memcpy(&hP, h + 28, 4);
  memcpy(&kind, h + 32, 4);
  memcpy(&sep, h + 36, 4);
  memcpy(&vocab, h + 40, 4);
  memcpy(&n_win, h + 44, 4);
  memcpy(&mcrc, h + 56, 4);
  uint64_t seed;
  memcpy(&seed, h + 48, 8);
  if (ver != kContainerVersion || hW != (uint32_t)W || hP != (uint32_t)c.cdf_bits || kind != (uint32_t)c.input_kind ||
      sep != serial_word(c) || vocab != (uint32_t)c.vocab || mcrc != model_crc(c) || seed != c.weight_seed)
    return fail(ctx, LMGC_ERR_CORRUPT, "container does not match this context's model or coder");
  if ((uint64_t)n_win != (n_tok + W - 1) / W || 64 + 8 * (size_t)n_win > in_bytes)
    return fail(ctx, LMGC_ERR_CORRUPT, "container window table truncated");
  if (cap_tok < n_ids * (size_t)W) return fail(ctx, LMGC_ERR_NO_SPACE, "token buffer too small");
  std::vector<uint32_t> bl(n_win), crc_tab(n_win);
  if (n_win) {
    LMGC_CUDA(ctx, cudaMemcpy(bl.data(), d_in + 64, 4 * (size_t)n_win, cudaMemcpyDeviceToHost));
    LMGC_CUDA(ctx, cudaMemcpy(crc_tab.data(), d_in + 64 + 4 * (size_t)n_win, 4 * (size_t)n_win,
                              cudaMemcpyDeviceToHost));
  }
  std::vector<uint64_t> off(n_win + 1);
  off[0] = 64 + 8 * (uint64_t)n_win;
  for (uint32_t w = 0; w < n_win; w++) off[w + 1] = off[w] + (bl[w] + 7) / 8;
  if (off[n_win] > in_bytes) return fail(ctx, LMGC_ERR_CORRUPT, "container payload truncated");
  for (size_t i = 0; i < n_ids; i++)
    if (h_win_ids[i] >= n_win) return fail(ctx, LMGC_ERR_INVALID, "window id out of range");
  const size_t kv_per_win = decode_kv_per_window(ctx);
  // decode batch: as many of the requested windows as a KV cache of half the free device memory
  // holds -- a step's GEMMs cost about the same for 64 rows as for 256
  size_t batch = 0;
  LMGC_CUDA(ctx, decode_batch(ctx, &batch));
  const int64_t nd_max = std::max<int64_t>(1, std::min<int64_t>((int64_t)std::max<size_t>(n_ids, 1), (int64_t)batch));
  const size_t kv_need = kv_per_win * (size_t)nd_max;
  if (ctx->kv_cap < kv_need || !ctx->kv_cache) {
    LMGC_CUDA(ctx, ensure(&ctx->kv_cache, &ctx->kv_cap, kv_need));
    // keys/values past a decoded position are read (and multiplied by probability 0): keep them finite
    LMGC_CUDA(ctx, cudaMemsetAsync(ctx->kv_cache, 0, ctx->kv_cap, s));
  }
  // per-chunk device arrays: code offsets, bit lengths, lengths, decoder states
  void* dev = nullptr;
  const size_t st_bytes = dec_state_bytes();
  const size_t arr = (size_t)nd_max * (8 + 4 + 4 + 4) + (size_t)nd_max * st_bytes + 256;
  LMGC_CUDA(ctx, cudaMallocAsync(&dev, arr, s));
  uint64_t* d_coff = (uint64_t*)dev;
  uint32_t* d_bl = (uint32_t*)(d_coff + nd_max);
  uint32_t* d_len = d_bl + nd_max;
  uint32_t* d_crc = d_len + nd_max;
  void* d_state = (void*)(((uintptr_t)(d_crc + nd_max) + 63) / 64 * 64);
  lmgc_status st = LMGC_OK;
  for (size_t i0 = 0; i0 < n_ids && st == LMGC_OK; i0 += nd_max) {
    const int64_t nd = std::min<int64_t>(nd_max, (int64_t)(n_ids - i0));
    std::vector<uint64_t> hoff(nd);
    std::vector<uint32_t> hbl(nd), hlen(nd);
    int64_t max_len = 0;
    for (int64_t j = 0; j < nd; j++) {
      uint32_t w = h_win_ids[i0 + j];
      hoff[j] = off[w];
      hbl[j] = bl[w];
      hlen[j] = (uint32_t)std::min<uint64_t>((uint64_t)W, n_tok - (uint64_t)w * W);
      max_len = std::max<int64_t>(max_len, hlen[j]);
    }
    cudaMemcpyAsync(d_coff, hoff.data(), 8 * nd, cudaMemcpyHostToDevice, s);
    cudaMemcpyAsync(d_bl, hbl.data(), 4 * nd, cudaMemcpyHostToDevice, s);
    cudaMemcpyAsync(d_len, hlen.data(), 4 * nd, cudaMemcpyHostToDevice, s);
    launch_dec_init(d_in, d_coff, d_bl, nd, d_state, s);
    uint16_t* out = d_tok + i0 * W;
    for (int64_t pos = 0; pos < max_len; pos++) {
      note_launch();
      k_dec_inputs<<<(unsigned)((nd + 127) / 128), 128, 0, s>>>(out, nd, W, pos, ctx->ws.tok_in);
      embed_rows(ctx, nd, s);
      forward_layers(ctx, nd, nd, true, pos, s, c.alphabet != 0);
      if (c.alphabet)
        launch_dec_search_alpha(ctx->logits, nd, kAlphaCols, c.cdf_bits, ctx->exp2_tab, d_state, d_in, out, W, pos,
                                d_len, ctx->alpha_cols, ctx->d_err, s);
      else
        launch_dec_search(ctx->logits, nd, c.vocab, c.cdf_bits, ctx->exp2_tab, d_state, d_in, out, W, pos, d_len,
                          ctx->d_err, s);
    }
    // every restored window must reproduce the container's token checksum
    launch_window_crc(out, W, d_len, nd, d_crc, s);
    std::vector<uint32_t> got(nd);
    cudaMemcpyAsync(got.data(), d_crc, 4 * nd, cudaMemcpyDeviceToHost, s);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) st = cuda_fail(ctx, e, "decode");
    else st = check_err_word(ctx, s, "decode");
    for (int64_t j = 0; j < nd && st == LMGC_OK; j++)
      if (got[j] != crc_tab[h_win_ids[i0 + j]])
        st = fail(ctx, LMGC_ERR_CORRUPT, "decoded window does not match its token checksum");
  }
  cudaFreeAsync(dev, s);
  cudaStreamSynchronize(s);
  if (ctx->prof.enabled) prof_collect(ctx);
  return st;
}

lmgc_status lmgc_decode_batch_windows(lmgc_ctx* ctx, size_t* n) {
  if (!ctx || !n) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  LMGC_CUDA(ctx, decode_batch(ctx, n));
  return LMGC_OK;
}

lmgc_status lmgc_launch_count(uint64_t* n) {
  if (!n) return LMGC_ERR_INVALID;
  *n = g_launches.load(std::memory_order_relaxed);
  return LMGC_OK;
}

lmgc_status lmgc_gemm(lmgc_ctx* ctx, const void* d_a, const void* d_b, void* d_c, size_t M, size_t N, size_t K,
                      int epi, lmgc_stream stream) {
  if (!ctx || (M && N && (!d_a || !d_b || !d_c))) return fail(ctx, LMGC_ERR_INVALID, "null argument");
  if (K % 8 || epi < 0 || (epi > 3 && epi != kAddResidualWide))
    return fail(ctx, LMGC_ERR_INVALID, "lmgc_gemm: K must be a multiple of 8, epi 0..3 or 5");
  if (epi == kSwiGLU && !(ctx->cfg.dtype == LMGC_BF16 && tc_gemm_supported(M, N, K, epi)))
    return fail(ctx, LMGC_ERR_INVALID, "lmgc_gemm: epi 3 needs the bf16 tensor-core path and N % 256 == 0");
  if (ctx->cfg.dtype == LMGC_BF16 && M && N && !tc_gemm_supported(M, N, K, epi))
    return fail(ctx, LMGC_ERR_INVALID, "lmgc_gemm: shape outside the tcgen05 kernel");
  if (ctx->cfg.dtype != LMGC_BF16 && (epi == kSwiGLU || epi == kQKVRope))
    return fail(ctx, LMGC_ERR_INVALID, "lmgc_gemm: epilogue 3 is for bf16 models");
  // the operands are read by TMA, whose global addresses must be 16-byte aligned, and the
  // epilogues write C with 16-byte vector stores
  if (((uintptr_t)d_a | (uintptr_t)d_b | (uintptr_t)d_c) & 15)
    return fail(ctx, LMGC_ERR_INVALID, "lmgc_gemm: A, B and C must be 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  gemm(ctx, d_a, d_b, d_c, (int64_t)M, (int64_t)N, (int64_t)K, epi, s);
  LMGC_CUDA(ctx, cudaGetLastError());
  if (ctx->prof.enabled) {
    cudaStreamSynchronize(s);
    prof_collect(ctx);
  }
  return check_err_word(ctx, s, "gemm");
}

lmgc_status lmgc_stage_times(const lmgc_ctx* ctx, float* ms, size_t n_ms) {
  if (!ctx || !ms) return LMGC_ERR_INVALID;
  for (size_t i = 0; i < n_ms && i < 5; i++) ms[i] = ctx->stage_ms[i];
  return LMGC_OK;
}

lmgc_status lmgc_profile(lmgc_ctx* ctx, int enable) {
  if (!ctx) ctx = free_ctx();
  ctx->prof.enabled = enable != 0;
  for (int i = 0; i < kNumClasses; i++) ctx->prof.stats[i] = KernelStat{kClassNames[i], 0, 0.f, 0.0};
  return LMGC_OK;
}

lmgc_status lmgc_kernel_stats(const lmgc_ctx* ctx, int cls, char* name, size_t name_len, int* launches, float* ms,
                              double* work) {
  if (!ctx) ctx = free_ctx();
  if (cls < 0 || cls >= kNumClasses) return LMGC_ERR_INVALID;
  const KernelStat& st = ctx->prof.stats[cls];
  if (name && name_len) {
    size_t n = std::min(name_len - 1, strlen(kClassNames[cls]));
    memcpy(name, kClassNames[cls], n);
    name[n] = 0;
  }
  if (launches) *launches = st.launches;
  if (ms) *ms = st.ms;
  if (work) *work = st.work;
  return LMGC_OK;
}

}  // extern "C"
