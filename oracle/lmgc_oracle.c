/*
 * lmgc_oracle.c -- plain, slow CPU oracle for the LM-GC encode path
 * ("Language Models as Zero-shot Lossless Gradient Compressors", arXiv 2409.17836).
 *
 * TEST INFRASTRUCTURE ONLY. Only the tests, the package smoke check and the bench's
 * CPU-baseline leg may load this library. It shares no code, header, table or constant
 * generator with the CUDA path, and it never calls into it.
 *
 * What it computes, step by step, and the passage each step follows:
 *   serialisation ........ Sec. 4 "Serialization" and Fig. 1: every 4 bits of an fp32 become
 *                          one hex digit, 8 digits per value, then a separator.
 *   windows + BOS ........ Sec. 4 "Compression", Eq. 2: p(t_k | BOS, t_<k); BOS is context
 *                          only; decoding runs until the window is full.
 *   LM prior ............. Eq. 1 / Eq. 2 with a Llama-family decoder (Sec. 5.1 names
 *                          TinyLlama / OpenLLaMA / Llama 2), fp64 arithmetic.
 *   integer CDF .......... implied by the Torchac-based coder of Sec. 5.1 (integer CDFs)
 *                          (Sec. 5.1 "Implementation"): an integer-exact quantiser.
 *   arithmetic coder ..... Sec. 3 "Arithmetic coding" (interval subdivision, any number of
 *                          the final interval represents the message) in an exact integer form.
 *
 * Readings where the paper is silent are the ones listed in the design notes of the
 * repository (MSB-first nibbles, character-level token ids, the quantiser, the coder's
 * termination). Parity of the LM logits is pinned only through invariants and library
 * routines (causality, zero weights, RMSNorm / attention / SiLU against torch), not
 * against printed values: the paper prints none.
 *
 * Build: gcc -O2 -std=c11 -fPIC -shared -ffp-contract=off -fopenmp -o liblmgc_oracle.so
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "exp2_tables.h"

#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------------------------ */
/* Token alphabet (reading of Sec. 4 / Fig. 1 with a character-level tokeniser):              */
/* hex digit v -> id v (0..15); ' ' -> 16, ',' -> 17, ';' -> 18; BOS -> 19.                  */
/* ------------------------------------------------------------------------------------------ */
#define ORC_TOK_SPACE 16
#define ORC_TOK_COMMA 17
#define ORC_TOK_SEMI 18
#define ORC_TOK_BOS 19

/* Separator sequence for a separator mode (Table 1 variants H_s, H_c, H_{c+s}, H_semi, H_n). */
static int orc_sep_tokens(int sep_mode, uint16_t sep[2]) {
  switch (sep_mode) {
    case 0: sep[0] = ORC_TOK_SPACE; return 1;                        /* H_s     */
    case 1: sep[0] = ORC_TOK_COMMA; return 1;                        /* H_c     */
    case 2: sep[0] = ORC_TOK_COMMA; sep[1] = ORC_TOK_SPACE; return 2; /* H_{c+s} */
    case 3: sep[0] = ORC_TOK_SEMI; return 1;                         /* H_semi  */
    case 4: return 0;                                                /* H_n     */
    default: return -1;
  }
}

/* Hex digits per value: 8 for an fp32 value (4 bytes), 2 for a uint8 code (Sec. 5.4 Eq. 4). */
static int orc_digits(int input_kind) { return input_kind == 0 ? 8 : (input_kind == 1 ? 2 : -1); }

int64_t orc_tokens_per_value(int input_kind, int sep_mode) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep), nd = orc_digits(input_kind);
  if (ns < 0 || nd < 0) return -1;
  return nd + ns;
}

/* Sec. 4 "Serialization": the bits of each value, split into 4-bit groups, most significant
 * group first (sign and exponent first), each group one hex digit, then the separator. */
int64_t orc_serialize(int input_kind, int sep_mode, const void* in, int64_t n, uint16_t* out) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep), nd = orc_digits(input_kind);
  if (ns < 0 || nd < 0 || n < 0) return -1;
  int64_t t = 0;
  for (int64_t i = 0; i < n; i++) {
    uint32_t b = input_kind == 0 ? ((const uint32_t*)in)[i] : ((const uint8_t*)in)[i];
    for (int j = 0; j < nd; j++) out[t++] = (uint16_t)((b >> (4 * (nd - 1 - j))) & 0xFu);
    for (int s = 0; s < ns; s++) out[t++] = sep[s];
  }
  return t;
}

/* Inverse of orc_serialize. Returns the number of values, or -1 if the token stream is not
 * a well-formed serialisation. */
int64_t orc_deserialize(int input_kind, int sep_mode, const uint16_t* tok, int64_t n_tok, void* out) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep), nd = orc_digits(input_kind);
  if (ns < 0 || nd < 0 || n_tok < 0) return -1;
  int64_t per = nd + ns;
  if (n_tok % per) return -1;
  int64_t n = n_tok / per;
  for (int64_t i = 0; i < n; i++) {
    uint32_t b = 0;
    for (int j = 0; j < nd; j++) {
      uint16_t d = tok[i * per + j];
      if (d > 15) return -1;
      b = (b << 4) | d;
    }
    for (int s = 0; s < ns; s++)
      if (tok[i * per + nd + s] != sep[s]) return -1;
    if (input_kind == 0) ((uint32_t*)out)[i] = b;
    else ((uint8_t*)out)[i] = (uint8_t)b;
  }
  return n;
}

/* Byte grouping (Sec. 5.3 "Byte grouping", Fig. 3: bytes per group BPG in {1, 2, 3, 4, 8} and
 * none). The values' bytes are taken in order -- an fp32 value's four bytes most significant
 * first (order 0) or least significant first (order 1), a uint8 code as its one byte -- and each
 * byte becomes two hex digits, high nibble first. The separator follows every `group` bytes and
 * also the last group when it is partial. group 0 means one group per value, which is
 * orc_serialize's layout. Returns the token count of n values, or -1 for bad arguments. */
static int64_t orc_bytes_per_value(int input_kind) { return input_kind == 0 ? 4 : (input_kind == 1 ? 1 : -1); }

int64_t orc_serial_tokens(int input_kind, int sep_mode, int group, int order, int64_t n) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep);
  int64_t bv = orc_bytes_per_value(input_kind);
  if (ns < 0 || bv < 0 || group < 0 || group > 8 || order < 0 || order > 1 || n < 0) return -1;
  int64_t g = group ? group : bv, nbytes = n * bv;
  return 2 * nbytes + ns * ((nbytes + g - 1) / g);
}

/* byte j (0-based, in stream order) of value i */
static uint32_t orc_value_byte(int input_kind, int order, const void* in, int64_t i, int j) {
  if (input_kind == 1) return ((const uint8_t*)in)[i];
  uint32_t b = ((const uint32_t*)in)[i];
  int shift = order == 0 ? 8 * (3 - j) : 8 * j;
  return (b >> shift) & 0xFFu;
}

int64_t orc_serialize_grouped(int input_kind, int sep_mode, int group, int order, const void* in, int64_t n,
                              uint16_t* out) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep);
  if (orc_serial_tokens(input_kind, sep_mode, group, order, n) < 0) return -1;
  int64_t bv = orc_bytes_per_value(input_kind), g = group ? group : bv, nbytes = n * bv, t = 0;
  for (int64_t k = 0; k < nbytes; k++) {
    uint32_t byte = orc_value_byte(input_kind, order, in, k / bv, (int)(k % bv));
    out[t++] = (uint16_t)(byte >> 4);
    out[t++] = (uint16_t)(byte & 0xFu);
    if ((k + 1) % g == 0 || k + 1 == nbytes)
      for (int s = 0; s < ns; s++) out[t++] = sep[s];
  }
  return t;
}

/* Inverse of orc_serialize_grouped: the number of values, or -1 if no value count gives n_tok
 * tokens or a token is out of place. */
int64_t orc_deserialize_grouped(int input_kind, int sep_mode, int group, int order, const uint16_t* tok,
                                int64_t n_tok, void* out) {
  uint16_t sep[2];
  int ns = orc_sep_tokens(sep_mode, sep);
  if (orc_serial_tokens(input_kind, sep_mode, group, order, 0) < 0 || n_tok < 0) return -1;
  int64_t bv = orc_bytes_per_value(input_kind), g = group ? group : bv;
  /* the token count grows with n: find n by stepping (each value adds at least 2 tokens) */
  int64_t n = n_tok / (2 * bv + ns * bv);
  while (orc_serial_tokens(input_kind, sep_mode, group, order, n) < n_tok) n++;
  if (orc_serial_tokens(input_kind, sep_mode, group, order, n) != n_tok) return -1;
  int64_t nbytes = n * bv, t = 0;
  if (input_kind == 0) memset(out, 0, (size_t)n * 4);
  for (int64_t k = 0; k < nbytes; k++) {
    uint16_t hi = tok[t++], lo = tok[t++];
    if (hi > 15 || lo > 15) return -1;
    uint32_t byte = (uint32_t)(hi << 4 | lo);
    int64_t i = k / bv;
    int j = (int)(k % bv);
    if (input_kind == 1) {
      ((uint8_t*)out)[i] = (uint8_t)byte;
    } else {
      int shift = order == 0 ? 8 * (3 - j) : 8 * j;
      ((uint32_t*)out)[i] |= byte << shift;
    }
    if ((k + 1) % g == 0 || k + 1 == nbytes)
      for (int s = 0; s < ns; s++)
        if (tok[t++] != sep[s]) return -1;
  }
  return n;
}

/* ------------------------------------------------------------------------------------------ */
/* Random-init weights. The paper uses pretrained checkpoints (Sec. 5.1); they are absent, so  */
/* every weight is drawn from a counter-based generator: splitmix64 (Steele, Lea and Flood,    */
/* "Fast splittable pseudorandom number generators", OOPSLA 2014; the mixing function of       */
/* Vigna's splitmix64.c) applied to seed ^ (tensor_id << 40) ^ index. The top 24 bits u give  */
/* w = ((u - 2^23) * 2^-23) * a with a = fp32(init_std * sqrt(3)): uniform with std init_std. */
/* ------------------------------------------------------------------------------------------ */
uint64_t orc_splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* fp32 -> bf16 -> fp32 with round-to-nearest-even on the bit pattern (finite inputs). */
static float orc_round_bf16(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  u = u + 0x7FFFu + ((u >> 16) & 1u);
  u &= 0xFFFF0000u;
  float y;
  memcpy(&y, &u, 4);
  return y;
}

float orc_bf16_round(float x) { return orc_round_bf16(x); }

static float orc_scale(float init_std) { return (float)((double)init_std * sqrt(3.0)); }

float orc_weight(uint64_t seed, uint32_t tid, uint64_t idx, float init_std, int bf16) {
  uint64_t u = orc_splitmix64(seed ^ ((uint64_t)tid << 40) ^ idx) >> 40;
  float unit = (float)((int32_t)u - (1 << 23)) * (1.0f / 8388608.0f);
  float w = unit * orc_scale(init_std);
  return bf16 ? orc_round_bf16(w) : w;
}

void orc_weight_tensor(uint64_t seed, uint32_t tid, uint64_t n, float init_std, int bf16, float* out) {
  for (uint64_t i = 0; i < n; i++) out[i] = orc_weight(seed, tid, i, init_std, bf16);
}

/* ------------------------------------------------------------------------------------------ */
/* Model configuration (Llama family). Tensor ids: 0 = embedding E[V][d]; for layer l the ids  */
/* 1+7l .. 7+7l are Wq[nq*hd][d], Wk[nkv*hd][d], Wv[nkv*hd][d], Wo[d][nq*hd], Wgate[ffn][d],  */
/* Wup[ffn][d], Wdown[d][ffn]; 1+7L is the vocabulary head Wvocab[V][d]. Index = row-major.   */
/* ------------------------------------------------------------------------------------------ */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, d_ffn, vocab;
  int32_t bf16;      /* 1: weights rounded to bf16 (values exact; arithmetic stays fp64) */
  int32_t window;
  uint64_t weight_seed;
  float init_std, rms_eps, rope_theta;
  int32_t n_threads; /* OpenMP threads for the linear layers (1 = serial) */
  /* restricted-alphabet coding (0 ids: the whole vocabulary): the integer CDF of a position is
   * taken over the logits of these ids only (ascending), and the coded symbol is the token's
   * index among them */
  int32_t n_alpha;
  uint16_t alpha[32];
} orc_cfg;

/* sizeof(orc_cfg), and the offsets of its 14 fields in declaration order into off[0..13], so that
 * a binding can check its copy of the struct */
size_t orc_cfg_layout(size_t* off) {
  const size_t o[14] = {offsetof(orc_cfg, n_layers),   offsetof(orc_cfg, d_model),   offsetof(orc_cfg, n_heads),
                        offsetof(orc_cfg, n_kv_heads), offsetof(orc_cfg, d_ffn),     offsetof(orc_cfg, vocab),
                        offsetof(orc_cfg, bf16),       offsetof(orc_cfg, window),    offsetof(orc_cfg, weight_seed),
                        offsetof(orc_cfg, init_std),   offsetof(orc_cfg, rms_eps),   offsetof(orc_cfg, rope_theta),
                        offsetof(orc_cfg, n_threads),  offsetof(orc_cfg, n_alpha)};
  for (int i = 0; i < 14; i++) off[i] = o[i];
  return sizeof(orc_cfg);
}

enum { ORC_WQ = 0, ORC_WK, ORC_WV, ORC_WO, ORC_WGATE, ORC_WUP, ORC_WDOWN };

static uint32_t orc_tid_layer(int l, int which) { return (uint32_t)(1 + 7 * l + which); }
static uint32_t orc_tid_head(const orc_cfg* c) { return (uint32_t)(1 + 7 * c->n_layers); }

/* RMSNorm with unit gain: y = x / sqrt(mean(x^2) + eps). */
void orc_rmsnorm(const double* x, int64_t rows, int d, double eps, double* y) {
  for (int64_t r = 0; r < rows; r++) {
    double ss = 0.0;
    for (int j = 0; j < d; j++) ss += x[r * d + j] * x[r * d + j];
    double inv = 1.0 / sqrt(ss / d + eps);
    for (int j = 0; j < d; j++) y[r * d + j] = x[r * d + j] * inv;
  }
}

/* Rotary position embedding, rotate-half pairing: within each head, dims i and i + hd/2 are
 * rotated by angle pos * theta^(-2i/hd). x is [rows][n_heads*hd], pos[r] the position of row r. */
void orc_rope(double* x, int64_t rows, const int64_t* pos, int n_heads, int hd, double theta) {
  int half = hd / 2;
  for (int64_t r = 0; r < rows; r++)
    for (int h = 0; h < n_heads; h++) {
      double* v = x + r * (int64_t)n_heads * hd + (int64_t)h * hd;
      for (int i = 0; i < half; i++) {
        double ang = (double)pos[r] * pow(theta, -2.0 * i / hd);
        double c = cos(ang), s = sin(ang);
        double a = v[i], b = v[i + half];
        v[i] = a * c - b * s;
        v[i + half] = a * s + b * c;
      }
    }
}

/* Causal softmax attention of n_new query rows at positions p0..p0+n_new-1 against keys and
 * values at positions 0..p0+n_new-1. q is [n_new][nq*hd]; kc, vc are [>=p0+n_new][nkv*hd].
 * Query head h reads key/value head h / (nq/nkv) (grouped-query attention). Scale 1/sqrt(hd). */
void orc_attention(const double* q, const double* kc, const double* vc, int64_t p0, int64_t n_new,
                   int nq, int nkv, int hd, double* out) {
  int group = nq / nkv;
  double scale = 1.0 / sqrt((double)hd);
  double* s = (double*)malloc(sizeof(double) * (size_t)(p0 + n_new));
  for (int64_t r = 0; r < n_new; r++) {
    int64_t p = p0 + r;
    for (int h = 0; h < nq; h++) {
      int kh = h / group;
      const double* qv = q + r * (int64_t)nq * hd + (int64_t)h * hd;
      double m = -INFINITY;
      for (int64_t j = 0; j <= p; j++) {
        const double* kv = kc + j * (int64_t)nkv * hd + (int64_t)kh * hd;
        double dot = 0.0;
        for (int i = 0; i < hd; i++) dot += qv[i] * kv[i];
        s[j] = dot * scale;
        if (s[j] > m) m = s[j];
      }
      double sum = 0.0;
      for (int64_t j = 0; j <= p; j++) {
        s[j] = exp(s[j] - m);
        sum += s[j];
      }
      double* o = out + r * (int64_t)nq * hd + (int64_t)h * hd;
      for (int i = 0; i < hd; i++) o[i] = 0.0;
      for (int64_t j = 0; j <= p; j++) {
        const double* vv = vc + j * (int64_t)nkv * hd + (int64_t)kh * hd;
        double w = s[j] / sum;
        for (int i = 0; i < hd; i++) o[i] += w * vv[i];
      }
    }
  }
  free(s);
}

/* SiLU-gated MLP product: a = silu(g) * u, silu(x) = x / (1 + exp(-x)). */
void orc_swiglu(const double* g, const double* u, int64_t n, double* a) {
  for (int64_t i = 0; i < n; i++) a[i] = g[i] / (1.0 + exp(-g[i])) * u[i];
}

/* y[r][o] (+)= sum_i x[r][i] * W[o][i], W generated row by row from (seed, tid). */
static void orc_linear(const orc_cfg* c, uint32_t tid, const double* x, int64_t rows, int in, int outd,
                       double* y, int accumulate) {
#pragma omp parallel for schedule(static) num_threads(c->n_threads > 0 ? c->n_threads : 1) if (c->n_threads > 1)
  for (int o = 0; o < outd; o++) {
    double* w = (double*)malloc(sizeof(double) * (size_t)in);
    for (int i = 0; i < in; i++)
      w[i] = orc_weight(c->weight_seed, tid, (uint64_t)o * (uint64_t)in + (uint64_t)i, c->init_std, c->bf16);
    for (int64_t r = 0; r < rows; r++) {
      double acc = 0.0;
      const double* xr = x + r * in;
      for (int i = 0; i < in; i++) acc += xr[i] * w[i];
      if (accumulate) y[r * outd + o] += acc;
      else y[r * outd + o] = acc;
    }
    free(w);
  }
}

/* Incremental forward state of one window: the residual is recomputed per call, keys and
 * values of every layer are kept for all positions fed so far (the KV cache of Sec. 6). */
typedef struct {
  orc_cfg c;
  int64_t n_pos; /* positions already fed */
  int64_t max_pos;
  double* kc;    /* [n_layers][max_pos][nkv*hd] */
  double* vc;
} orc_lm;

orc_lm* orc_lm_new(const orc_cfg* c, int64_t max_pos) {
  orc_lm* s = (orc_lm*)calloc(1, sizeof(orc_lm));
  if (!s) return NULL;
  s->c = *c;
  s->max_pos = max_pos;
  int hd = c->d_model / c->n_heads;
  size_t kv = (size_t)c->n_layers * (size_t)max_pos * (size_t)c->n_kv_heads * (size_t)hd;
  s->kc = (double*)calloc(kv, sizeof(double));
  s->vc = (double*)calloc(kv, sizeof(double));
  if (!s->kc || !s->vc) {
    free(s->kc); free(s->vc); free(s);
    return NULL;
  }
  return s;
}

void orc_lm_free(orc_lm* s) {
  if (!s) return;
  free(s->kc);
  free(s->vc);
  free(s);
}

/* Feed n_new input tokens (the first fed token of a window is BOS) at the next positions and
 * write the next-token logits of each fed position: logits[r] = log-potentials of
 * p(t | BOS, t_<k) at position n_pos + r (Eq. 2). Returns 0, or -1 on bad arguments. */
int orc_lm_feed(orc_lm* s, const uint16_t* tok_in, int64_t n_new, double* logits) {
  const orc_cfg* c = &s->c;
  if (n_new <= 0 || s->n_pos + n_new > s->max_pos) return -1;
  int d = c->d_model, nq = c->n_heads, nkv = c->n_kv_heads, hd = d / nq, F = c->d_ffn, V = c->vocab;
  int64_t p0 = s->n_pos;
  double* x = (double*)malloc(sizeof(double) * (size_t)(n_new * d));
  double* n = (double*)malloc(sizeof(double) * (size_t)(n_new * d));
  double* q = (double*)malloc(sizeof(double) * (size_t)(n_new * nq * hd));
  double* k = (double*)malloc(sizeof(double) * (size_t)(n_new * nkv * hd));
  double* v = (double*)malloc(sizeof(double) * (size_t)(n_new * nkv * hd));
  double* o = (double*)malloc(sizeof(double) * (size_t)(n_new * nq * hd));
  double* g = (double*)malloc(sizeof(double) * (size_t)(n_new * F));
  double* u = (double*)malloc(sizeof(double) * (size_t)(n_new * F));
  int64_t* pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)n_new);
  for (int64_t r = 0; r < n_new; r++) {
    pos[r] = p0 + r;
    uint16_t t = tok_in[r];
    for (int j = 0; j < d; j++)
      x[r * d + j] = orc_weight(c->weight_seed, 0, (uint64_t)t * (uint64_t)d + (uint64_t)j, c->init_std, c->bf16);
  }
  for (int l = 0; l < c->n_layers; l++) {
    orc_rmsnorm(x, n_new, d, c->rms_eps, n);
    orc_linear(c, orc_tid_layer(l, ORC_WQ), n, n_new, d, nq * hd, q, 0);
    orc_linear(c, orc_tid_layer(l, ORC_WK), n, n_new, d, nkv * hd, k, 0);
    orc_linear(c, orc_tid_layer(l, ORC_WV), n, n_new, d, nkv * hd, v, 0);
    orc_rope(q, n_new, pos, nq, hd, c->rope_theta);
    orc_rope(k, n_new, pos, nkv, hd, c->rope_theta);
    double* kl = s->kc + (size_t)l * (size_t)s->max_pos * (size_t)(nkv * hd);
    double* vl = s->vc + (size_t)l * (size_t)s->max_pos * (size_t)(nkv * hd);
    memcpy(kl + p0 * nkv * hd, k, sizeof(double) * (size_t)(n_new * nkv * hd));
    memcpy(vl + p0 * nkv * hd, v, sizeof(double) * (size_t)(n_new * nkv * hd));
    orc_attention(q, kl, vl, p0, n_new, nq, nkv, hd, o);
    orc_linear(c, orc_tid_layer(l, ORC_WO), o, n_new, nq * hd, d, x, 1);
    orc_rmsnorm(x, n_new, d, c->rms_eps, n);
    orc_linear(c, orc_tid_layer(l, ORC_WGATE), n, n_new, d, F, g, 0);
    orc_linear(c, orc_tid_layer(l, ORC_WUP), n, n_new, d, F, u, 0);
    orc_swiglu(g, u, n_new * F, g);
    orc_linear(c, orc_tid_layer(l, ORC_WDOWN), g, n_new, F, d, x, 1);
  }
  orc_rmsnorm(x, n_new, d, c->rms_eps, n);
  orc_linear(c, orc_tid_head(c), n, n_new, d, V, logits, 0);
  s->n_pos += n_new;
  free(x); free(n); free(q); free(k); free(v); free(o); free(g); free(u); free(pos);
  return 0;
}

/* Logits of the first n_pos positions of one window whose tokens are win_tok[0..]:
 * the model input is [BOS, win_tok[0], ..., win_tok[n_pos-2]] (Eq. 2: BOS conditions the
 * first token and is never coded). */
int orc_lm_window_logits(const orc_cfg* c, const uint16_t* win_tok, int64_t n_pos, double* logits) {
  if (n_pos <= 0) return -1;
  orc_lm* s = orc_lm_new(c, n_pos);
  if (!s) return -1;
  uint16_t* in = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)n_pos);
  in[0] = ORC_TOK_BOS;
  for (int64_t i = 1; i < n_pos; i++) in[i] = win_tok[i - 1];
  int rc = orc_lm_feed(s, in, n_pos, logits);
  free(in);
  orc_lm_free(s);
  return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* Integer CDF (reading of the Torchac-based coder of Sec. 5.1; the paper does not say how    */
/* the LM probabilities were made integer). T = 2^P, row z[0..V) of fp32 logits:               */
/*  (i)   m = max z                                                                            */
/*  (ii)  y_j = fp32(fp32(z_j - m) * C), C = fp32(2^16 * log2 e)   (round to nearest, no FMA) */
/*  (iii) a_j = -rint(y_j) >= 0, clamped to 40 * 2^16 (y_j < -40 * 2^16 gives the cap directly) */
/*  (iv)  e_j = ((H[(a>>8)&255] * L[a&255] + 2^30) >> 31) >> (a >> 16)   ~ 2^31 * exp(z_j - m) */
/*  (v)   S = sum e_j                                                                          */
/*  (vi)  g_j = floor(e_j * (T - V) / S); freq_j = 1 + g_j; the residual (T - V) - sum g_j     */
/*        goes to the lowest index of the largest e_j                                          */
/*  (vii) cdf[0] = 0, cdf[j+1] = cdf[j] + freq_j, cdf[V] = T                                   */
/* ------------------------------------------------------------------------------------------ */
#define ORC_A_MAX (40LL * 65536LL)

void orc_exp2_tables(uint32_t* H, uint32_t* L) {
  memcpy(H, ORC_EXP2_H, sizeof(ORC_EXP2_H));
  memcpy(L, ORC_EXP2_L, sizeof(ORC_EXP2_L));
}

uint32_t orc_exp2_fixed(int64_t a) {
  if (a < 0) a = 0;
  if (a > ORC_A_MAX) a = ORC_A_MAX;
  uint64_t hl = (uint64_t)ORC_EXP2_H[(a >> 8) & 255] * (uint64_t)ORC_EXP2_L[a & 255];
  uint64_t e = (hl + (1ull << 30)) >> 31;
  return (uint32_t)(e >> (a >> 16));
}

static float orc_cdf_C(void) { return (float)(65536.0 * 1.4426950408889634073599246810019); }

/* Returns 0, or -1 if (V, P) is invalid (need 2 <= V < 2^P, P <= 31). */
int orc_quantize_cdf(const float* z, int V, int P, uint32_t* cdf) {
  if (V < 2 || P < 1 || P > 31 || (int64_t)V >= (1LL << P)) return -1;
  const uint64_t T = 1ull << P;
  const uint64_t M = T - (uint64_t)V;
  const float C = orc_cdf_C();
  float m = z[0];
  for (int j = 1; j < V; j++)
    if (z[j] > m) m = z[j];
  uint32_t* e = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)V);
  uint64_t S = 0;
  int amax = 0;
  for (int j = 0; j < V; j++) {
    float dz = z[j] - m;
    float y = dz * C;
    /* (iii) with the clamp applied before the conversion: y below -40*2^16 gives the cap */
    int64_t a = (y < -(float)ORC_A_MAX) ? ORC_A_MAX : -(int64_t)rintf(y);
    e[j] = orc_exp2_fixed(a);
    S += e[j];
    if (e[j] > e[amax]) amax = j;
  }
  uint64_t gsum = 0;
  cdf[0] = 0;
  for (int j = 0; j < V; j++) {
    uint64_t gj = ((uint64_t)e[j] * M) / S;
    gsum += gj;
    cdf[j + 1] = (uint32_t)(cdf[j] + 1 + gj);
  }
  uint64_t resid = M - gsum;
  for (int j = amax + 1; j <= V; j++) cdf[j] += (uint32_t)resid;
  free(e);
  return 0;
}

/* (start, freq) of symbol sym under the quantised CDF of row z. */
int orc_cdf_pair(const float* z, int V, int P, int sym, uint32_t* start, uint32_t* freq) {
  if (sym < 0 || sym >= V) return -1;
  uint32_t* cdf = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)(V + 1));
  int rc = orc_quantize_cdf(z, V, P, cdf);
  if (rc == 0) {
    *start = cdf[sym];
    *freq = cdf[sym + 1] - cdf[sym];
  }
  free(cdf);
  return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* Arithmetic coder (Sec. 3 "Arithmetic coding": the interval is split by P_AC per symbol,    */
/* symbol order low-to-high; any number of the final interval stands for the message).        */
/* Exact integer form: range R (62 bits), low L (unbounded), B = bits shifted so far.          */
/* Start R = 2^62, L = 0, B = 0. Per symbol (s = start, f = freq, T = 2^P):                    */
/*   r = R >> P;  L += r*s;  R = r*f;  k = max(0, 62 - bitlen(R));  R <<= k;  L <<= k;  B += k */
/* Termination: v = ceil(L / 2^60) * 2^60 lies in [L, L + R) since R >= 2^61; the code is the  */
/* top B + 2 bits of v as a (B + 62)-bit number, most significant bit first.                   */
/* Here L is held literally as one byte per bit, most significant first: bit index B + 61 is  */
/* L's least significant bit, "L <<= k" appends k zero bits, an addition carries towards 0.   */
/* ------------------------------------------------------------------------------------------ */
static int orc_bitlen64(uint64_t x) {
  int n = 0;
  while (x) {
    n++;
    x >>= 1;
  }
  return n;
}

/* Encodes n symbols. Writes ceil(l/8) bytes (MSB-first, zero padded) to out when it fits in
 * cap_bytes. Returns the bit length l, -1 on a bad argument, or -(l + 2) when out is too small
 * (so the caller learns l either way). */
int64_t orc_range_encode(const uint32_t* start, const uint32_t* freq, int64_t n, int P, uint8_t* out,
                         int64_t cap_bytes) {
  if (P < 1 || P > 31 || n < 0) return -1;
  const uint64_t T = 1ull << P;
  int64_t nbits_cap = n * (int64_t)P + 64 + 2;
  uint8_t* bit = (uint8_t*)calloc((size_t)nbits_cap, 1);
  if (!bit) return -1;
  uint64_t R = 1ull << 62;
  int64_t B = 0;
  for (int64_t i = 0; i < n; i++) {
    uint64_t s = start[i], f = freq[i];
    if (f == 0 || s + f > T) {
      free(bit);
      return -1;
    }
    uint64_t r = R >> P;
    uint64_t c = r * s; /* < 2^62 */
    /* L += c: add c's 62 bits at indices B+61 (lsb) .. B (bit 61 of c), carry toward 0 */
    int carry = 0;
    for (int b = 0; b < 62; b++) {
      int64_t idx = B + 61 - b;
      int sum = bit[idx] + (int)((c >> b) & 1u) + carry;
      bit[idx] = (uint8_t)(sum & 1);
      carry = sum >> 1;
    }
    for (int64_t idx = B - 1; carry && idx >= 0; idx--) {
      int sum = bit[idx] + carry;
      bit[idx] = (uint8_t)(sum & 1);
      carry = sum >> 1;
    }
    R = r * f;
    int k = 62 - orc_bitlen64(R);
    if (k < 0) k = 0;
    R <<= k;
    B += k; /* L <<= k: k zero bits appended below */
  }
  /* v = ceil(L / 2^60) * 2^60: add one at index B+1 if any of the 60 low bits is set */
  int any = 0;
  for (int64_t idx = B + 2; idx < B + 62; idx++) any |= bit[idx];
  if (any) {
    int carry = 1;
    for (int64_t idx = B + 1; carry && idx >= 0; idx--) {
      int sum = bit[idx] + carry;
      bit[idx] = (uint8_t)(sum & 1);
      carry = sum >> 1;
    }
  }
  int64_t len = B + 2;
  int64_t nbytes = (len + 7) / 8;
  if (nbytes > cap_bytes) {
    free(bit);
    return -(len + 2);
  }
  for (int64_t i = 0; i < nbytes; i++) {
    uint8_t byte = 0;
    for (int j = 0; j < 8; j++) {
      int64_t idx = i * 8 + j;
      byte = (uint8_t)((byte << 1) | (idx < len ? bit[idx] : 0));
    }
    out[i] = byte;
  }
  free(bit);
  return len;
}

/* Decoder (Sec. 3: decoding walks the same interval subdivision, finding at each step the
 * symbol whose interval holds the code). D = first 62 bits of the code (zero padded). Per symbol: r = R >> P;
 * t = D / r (t >= T means a corrupt code); s with cdf[s] <= t < cdf[s+1]; D -= r * cdf[s];
 * R = r * f_s; renormalise by the same k as the encoder, shifting the next k code bits into D. */
typedef struct {
  const uint8_t* in;
  int64_t nbits;
  int64_t pos;
  uint64_t R, D;
} orc_dec;

static int orc_dec_bit(orc_dec* d) {
  int v = 0;
  if (d->pos < d->nbits) v = (d->in[d->pos >> 3] >> (7 - (d->pos & 7))) & 1;
  d->pos++;
  return v;
}

void orc_dec_init(orc_dec* d, const uint8_t* in, int64_t nbits) {
  d->in = in;
  d->nbits = nbits;
  d->pos = 0;
  d->R = 1ull << 62;
  d->D = 0;
  for (int i = 0; i < 62; i++) d->D = (d->D << 1) | (uint64_t)orc_dec_bit(d);
}

int64_t orc_dec_size(void) { return (int64_t)sizeof(orc_dec); }

/* Returns the decoded symbol, or -1 if the code is corrupt. */
int orc_dec_step(orc_dec* d, const uint32_t* cdf, int V, int P) {
  uint64_t r = d->R >> P;
  uint64_t t = d->D / r;
  if (t >= (1ull << P)) return -1;
  int s = -1;
  for (int j = 0; j < V; j++)
    if (cdf[j] <= t && t < cdf[j + 1]) {
      s = j;
      break;
    }
  if (s < 0) return -1;
  d->D -= r * cdf[s];
  d->R = r * (uint64_t)(cdf[s + 1] - cdf[s]);
  int k = 62 - orc_bitlen64(d->R);
  if (k < 0) k = 0;
  for (int i = 0; i < k; i++) d->D = (d->D << 1) | (uint64_t)orc_dec_bit(d);
  d->R <<= k;
  return s;
}

/* ------------------------------------------------------------------------------------------ */
/* Whole windows: LM forward -> fp32 logits -> integer CDF -> (start, freq) -> one code per    */
/* window (Sec. 4 "Compression": windows are coded independently, each from a fresh BOS).     */
/* ------------------------------------------------------------------------------------------ */

/* The integer CDF of one position: over the whole vocabulary, or over the restricted alphabet
 * (the fp32 logits of its ids, in ascending id order). Returns the symbol count, or -1. */
static int orc_position_cdf(const orc_cfg* c, const float* z, int P, float* zs, uint32_t* cdf) {
  if (c->n_alpha <= 0) return orc_quantize_cdf(z, c->vocab, P, cdf) == 0 ? c->vocab : -1;
  for (int j = 0; j < c->n_alpha; j++) zs[j] = z[c->alpha[j]];
  return orc_quantize_cdf(zs, c->n_alpha, P, cdf) == 0 ? c->n_alpha : -1;
}

/* the coded symbol of token t: t itself, or its index in the restricted alphabet (-1: absent) */
static int orc_symbol(const orc_cfg* c, uint16_t t) {
  if (c->n_alpha <= 0) return t < c->vocab ? t : -1;
  for (int j = 0; j < c->n_alpha; j++)
    if (c->alpha[j] == t) return j;
  return -1;
}

/* (start, freq) pairs of one window's n tokens, from the oracle LM. pairs_start/freq: [n]. */
int orc_window_pairs(const orc_cfg* c, int P, const uint16_t* win_tok, int64_t n, uint32_t* pst, uint32_t* pfr,
                     float* logits_out /* optional [n][V] fp32 */) {
  int V = c->vocab;
  double* lg = (double*)malloc(sizeof(double) * (size_t)(n * V));
  float* z = (float*)malloc(sizeof(float) * (size_t)V);
  float zs[32];
  uint32_t* cdf = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)(V + 1));
  int rc = orc_lm_window_logits(c, win_tok, n, lg);
  for (int64_t i = 0; rc == 0 && i < n; i++) {
    for (int j = 0; j < V; j++) z[j] = (float)lg[i * V + j];
    if (logits_out) memcpy(logits_out + i * V, z, sizeof(float) * (size_t)V);
    const int sym = orc_symbol(c, win_tok[i]);
    if (orc_position_cdf(c, z, P, zs, cdf) < 0 || sym < 0) {
      rc = -1;
    } else {
      pst[i] = cdf[sym];
      pfr[i] = cdf[sym + 1] - cdf[sym];
    }
  }
  free(lg);
  free(z);
  free(cdf);
  return rc;
}

/* Encode windows [w0, w0 + nw) of a token stream of n_tok tokens (window length c->window).
 * Window w's code goes to out + w_local * cap_per_win; bitlen[w_local] gets its length.
 * Windows run in parallel over n_par OpenMP threads (the LM inside each is serial then).
 * Returns 0 or -1. */
int orc_encode_windows(const orc_cfg* c, int P, const uint16_t* tok, int64_t n_tok, int64_t w0, int64_t nw,
                       uint8_t* out, int64_t cap_per_win, int64_t* bitlen, int n_par) {
  int64_t W = c->window;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_par > 0 ? n_par : 1) if (n_par > 1) reduction(| : bad)
  for (int64_t wl = 0; wl < nw; wl++) {
    int64_t w = w0 + wl;
    int64_t b = w * W;
    int64_t n = n_tok - b < W ? n_tok - b : W;
    if (n <= 0) {
      bad |= 1;
      continue;
    }
    orc_cfg cc = *c;
    if (n_par > 1) cc.n_threads = 1;
    uint32_t* ps = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)n);
    uint32_t* pf = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)n);
    if (orc_window_pairs(&cc, P, tok + b, n, ps, pf, NULL) != 0) bad |= 1;
    else {
      int64_t len = orc_range_encode(ps, pf, n, P, out + wl * cap_per_win, cap_per_win);
      if (len < 0) bad |= 1;
      bitlen[wl] = len;
    }
    free(ps);
    free(pf);
  }
  return bad ? -1 : 0;
}

/* Decode one window of n tokens from its code (KV-cached: one LM position per step, each
 * step's logits quantised exactly as in encoding). Returns 0, or -1 if the code is corrupt. */
int orc_decode_window(const orc_cfg* c, int P, const uint8_t* code, int64_t nbits, int64_t n, uint16_t* tok_out) {
  int V = c->vocab;
  orc_lm* s = orc_lm_new(c, n);
  if (!s) return -1;
  double* lg = (double*)malloc(sizeof(double) * (size_t)V);
  float* z = (float*)malloc(sizeof(float) * (size_t)V);
  uint32_t* cdf = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)(V + 1));
  float zs[32];
  orc_dec d;
  orc_dec_init(&d, code, nbits);
  uint16_t cur = ORC_TOK_BOS;
  int rc = 0;
  for (int64_t i = 0; i < n && rc == 0; i++) {
    rc = orc_lm_feed(s, &cur, 1, lg);
    if (rc) break;
    for (int j = 0; j < V; j++) z[j] = (float)lg[j];
    const int nsym = orc_position_cdf(c, z, P, zs, cdf);
    if (nsym < 0) {
      rc = -1;
      break;
    }
    int sym = orc_dec_step(&d, cdf, nsym, P);
    if (sym < 0) {
      rc = -1;
      break;
    }
    const uint16_t t = c->n_alpha > 0 ? c->alpha[sym] : (uint16_t)sym;
    tok_out[i] = t;
    cur = t;
  }
  free(lg);
  free(z);
  free(cdf);
  orc_lm_free(s);
  return rc;
}

/* CRC-32 (IEEE 802.3, reflected polynomial 0xEDB88320, init and final xor 0xFFFFFFFF),
 * bit by bit. Used for the container header check. */
uint32_t orc_crc32(const uint8_t* p, int64_t n) {
  uint32_t c = 0xFFFFFFFFu;
  for (int64_t i = 0; i < n; i++) {
    c ^= p[i];
    for (int k = 0; k < 8; k++) c = (c >> 1) ^ (0xEDB88320u & (0u - (c & 1u)));
  }
  return c ^ 0xFFFFFFFFu;
}

int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
