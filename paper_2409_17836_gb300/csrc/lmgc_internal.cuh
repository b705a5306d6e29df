// lmgc_internal.cuh -- declarations shared by the .cu files of liblmgc.so (the CUDA path only).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/lmgc.h"

namespace lmgc {

// Token ids (character-level reading of Sec. 4 / Fig. 1).
constexpr int kTokSpace = 16, kTokComma = 17, kTokSemi = 18, kTokBos = 19;

// Device error word bits (set by bounded device loops instead of spinning or trapping).
enum : uint32_t { kErrCorrupt = 1u, kErrLimit = 2u, kErrDeser = 4u };

struct KernelStat {
  const char* name;
  int launches;
  float ms;
  double work;  // algorithmic flops or bytes summed over launches
};

// Timing of one kernel class inside a call (only when profiling is enabled).
struct Profiler {
  bool enabled = false;
  struct Rec {
    int cls;
    cudaEvent_t a, b;
    double work;
  };
  std::vector<Rec> pending;
  std::vector<cudaEvent_t> pool;
  KernelStat stats[16];
};

struct Layer {
  void* wqkv;   // [qkv_dim][d]: Wq rows, then Wk rows, then Wv rows
  void* wo;     // [d][nq*hd]
  void* wgu;    // [2*ffn][d]: gate/up rows, layout per GemmEpi::kSwiGLU
  void* wdown;  // [d][ffn]
};

struct Workspace {
  int64_t rows = 0;  // capacity in model rows (windows * W)
  float* x = nullptr;      // residual fp32 [rows][d]
  void* n = nullptr;       // normalised activations [rows][d] (T)
  void* qkv = nullptr;     // [rows][qkv_dim] (T)
  void* att = nullptr;     // [rows][nq*hd] (T)
  void* act = nullptr;     // SwiGLU output [rows][ffn] (T)
  void* gu = nullptr;      // gate/up GEMM output [rows][2*ffn] (T), unfused path only
  float* ss = nullptr;     // fused RMSNorm: per-row partial sums of squares [rows][d/256]
  uint16_t* tok_in = nullptr;  // model input ids [rows]
};

// Columns of the restricted alphabet's logits rows (its ids, then zero-weight padding).
constexpr int kAlphaCols = 32;

// The restricted alphabet: ids id[0..n) ascending, 2 <= n <= 32, each < vocab.
struct AlphaIds {
  int32_t n;
  int32_t id[32];
};

}  // namespace lmgc

struct lmgc_ctx {
  lmgc_config cfg;
  int device = 0;
  int hd = 0, qkv_dim = 0, tpv = 0;
  int kv_dim = 0;  // 2 n_kv_heads hd: a KV-cache row (keys, then values)
  size_t elt = 4;  // bytes per weight / activation element
  void* w_embed = nullptr;
  void* w_head = nullptr;
  std::vector<lmgc::Layer> layers;
  void* weights_blob = nullptr;
  float2* rope_cs = nullptr;   // [W][hd/2] (cos, sin)
  uint32_t* exp2_tab = nullptr;  // [512]: H then L
  lmgc::Workspace ws;
  float* logits = nullptr;     // [rows][V]
  // [rows]: order-preserving key of each logits row's maximum, written by the vocabulary GEMM of
  // a prefill (row_max_valid) and read by the CDF kernel in place of its max pass
  uint32_t* row_max = nullptr;
  bool row_max_valid = false;
  uint32_t* d_err = nullptr;   // device error word
  // encode staging
  uint16_t* tok = nullptr;
  size_t tok_cap = 0;
  uint32_t* pair_start = nullptr;
  uint32_t* pair_freq = nullptr;
  size_t pair_cap = 0;
  uint32_t* win_len = nullptr;
  size_t win_cap = 0;
  void* host_in = nullptr;  // device staging for lmgc_encode_host
  size_t host_in_cap = 0;
  uint8_t* host_out = nullptr;
  size_t host_out_cap = 0;
  // decode state
  void* kv_cache = nullptr;
  size_t kv_cap = 0;
  // codes of the last encode (slot scratch inside win_len)
  uint32_t* enc_bl = nullptr;
  uint32_t* enc_crc = nullptr;
  uint64_t* enc_off = nullptr;
  uint8_t* enc_slots = nullptr;
  size_t enc_slot = 0;
  int64_t enc_nwin = 0, enc_batches = 0;
  float stage_ms[5] = {0, 0, 0, 0, 0};
  cudaEvent_t ev[6] = {};
  std::vector<cudaEvent_t> batch_ev;
  lmgc::Profiler prof;
  bool fused_swiglu = false;  // gate/up interleaved, SwiGLU in the tcgen05 epilogue
  bool fused_rope = false;    // RoPE in the QKV tcgen05 epilogue
  bool fused_norm = false;    // RMSNorm folded into the GEMM epilogues (row scale + residual side outputs)
  lmgc::AlphaIds alpha{};     // cfg.alphabet == 1: the ids the serialisation can emit
  lmgc::AlphaIds alpha_cols{};  // the same as columns 0..n-1 of the narrow logits rows
  void* w_head_alpha = nullptr;  // [kAlphaCols][d]: alpha's rows of w_head, then zero rows
  std::string err;
};

namespace lmgc {

// ---- error helpers (host) ----
void set_thread_error(const std::string& s);
lmgc_status fail(lmgc_ctx* ctx, lmgc_status st, const std::string& msg);
lmgc_status cuda_fail(lmgc_ctx* ctx, cudaError_t e, const char* what);

#define LMGC_CUDA(ctx, call)                                   \
  do {                                                         \
    cudaError_t e_ = (call);                                   \
    if (e_ != cudaSuccess) return lmgc::cuda_fail(ctx, e_, #call); \
  } while (0)

// Counts kernel launches of this library (every launcher calls it once per launch).
void note_launch();

// ---- kernels' launchers (stream-ordered, no sync) ----
// serialize.cu
int tokens_per_value(int input_kind, int sep_mode);
// Byte grouping (Sec. 5.3): tokens of n values; the n with that many tokens (or -1); whether the
// layout is the default one group per value, most significant byte first.
int64_t serial_tokens(int input_kind, int sep_mode, int byte_group, int64_t n);
int64_t serial_values(int input_kind, int sep_mode, int byte_group, int64_t n_tok);
bool serial_is_default(int input_kind, int byte_group, int byte_order);
void launch_serialize(int input_kind, int sep_mode, int byte_group, int byte_order, const void* in, int64_t n,
                      uint16_t* tok, cudaStream_t s);
void launch_deserialize(int input_kind, int sep_mode, int byte_group, int byte_order, const uint16_t* tok,
                        int64_t n_values, void* out, uint32_t* err, cudaStream_t s);

// lm.cu
// Canonical row r of tensor tid goes to dst row row_off + (r / rblk) * rstride + r % rblk
// (rblk <= 0: dst row row_off + r).
void launch_init_weights(void* dst, int dtype, uint64_t seed, uint32_t tid, int64_t rows, int64_t cols, int64_t ld,
                         int64_t row_off, float init_std, cudaStream_t s, int64_t rblk = 0, int64_t rstride = 0);
void launch_window_inputs(const uint16_t* tok, int64_t n_tok, int64_t first_win, int64_t n_win, int W,
                          uint16_t* tok_in, cudaStream_t s);
void launch_embed(const uint16_t* tok_in, int64_t rows, const void* E, int d, int dtype, float* x, cudaStream_t s);
void launch_rmsnorm(const float* x, int64_t rows, int d, float eps, void* out, int dtype, cudaStream_t s);
// C[M][N] = A[M][K] . B[N][K]^T with the given epilogue
// kSwiGLU: B's rows are gate/up blocks interleaved 128 by 128 (rows 256t..256t+127 = gate rows
// 128t.., rows 256t+128.. = up rows 128t..); C[m][128t + j] = silu(gate) * up, N/2 columns.
// kQKVRope: kStore with the rotary embedding applied to the q and k heads (RopeArgs).
// kAddResidualWide: kAddResidual with 8 epilogue warps, each over half of a tile's columns, so
// its sums of squares come in 128-column parts (for short-K GEMMs whose epilogue would outlast
// the main loop).
enum GemmEpi { kStore = 0, kAddResidual = 1, kStoreF32 = 2, kSwiGLU = 3, kQKVRope = 4, kAddResidualWide = 5 };
// Fused RMSNorm (see gemm_tc.cu Params): consumers read row_ss (parts per row), residual
// producers write xh and ss_out.
struct NormArgs {
  const float* row_ss;
  int parts;
  float inv_d, eps;
  __half* xh;
  float* ss_out;
  uint32_t* row_max = nullptr;  // kStoreF32: atomic max of float_key(row values); zeroed by the caller
};
// Order-preserving map of fp32 (not NaN) to u32: a < b  <=>  float_key(a) < float_key(b); 0 is
// below every key, so a zeroed buffer is the identity of the max.
__host__ __device__ __forceinline__ uint32_t float_key(uint32_t bits) {
  return (bits & 0x80000000u) ? ~bits : (bits | 0x80000000u);
}
__host__ __device__ __forceinline__ uint32_t key_float_bits(uint32_t key) {
  return (key & 0x80000000u) ? (key & 0x7fffffffu) : ~key;
}
struct RopeArgs {
  const float2* cs;  // [W][hd/2] (cos, sin)
  int cols;          // columns [0, cols) are rotated: (n_heads + n_kv_heads) * hd
  int hd;
  int pos_mod;       // row m sits at position pos0 + m % pos_mod
  int64_t pos0;
};
// fp32 models: C (op)= A . B^T on the tensor cores in three-pass TF32 form (gemm_tf32.cu);
// epi kStore / kStoreF32 (C = acc) or kAddResidual (C += acc), C fp32 [M][N]
bool tf32_gemm_supported(int64_t M, int64_t N, int64_t K);
void launch_gemm_tf32(const float* A, const float* B, float* C, int64_t M, int64_t N, int64_t K, int epi,
                      uint32_t* err, cudaStream_t s);
void launch_rope(void* qkv, int64_t rows, int qkv_dim, int n_rot_heads, int hd, const float2* cs, int W,
                 int64_t pos_first, int64_t q_win_stride, int n_pos, int dtype, cudaStream_t s);
// fp32 models: causal attention on the tensor cores in three-pass TF32 form (attn_tf32.cu), head
// dim 32 or 64; arguments as launch_attention_tc's
bool tf32_attention_supported(int hd, int64_t q_dim, int64_t kv_dim);
void launch_attention_tf32(const float* q, int64_t q_rows, int64_t q_dim, const float* kv, int64_t kv_rows,
                           int64_t kv_dim, int k_off, int v_off, float* out, int64_t out_stride, int nq, int nkv,
                           int hd, int W, int64_t n_win, int64_t pos_first, int n_pos, int64_t q_win_stride,
                           uint32_t* err, cudaStream_t s);
void launch_swiglu(const void* gu, int64_t rows, int ffn, void* act, int dtype, cudaStream_t s);
void launch_copy_rows(const void* src, int64_t src_stride, void* dst, int64_t dst_win_stride, int64_t dst_pos,
                      int64_t n_rows, int64_t row_elems, int dtype, cudaStream_t s);

// cdf.cu
void upload_exp2_tables(uint32_t* d_tab, cudaStream_t s);  // builds H and L on the host
// mode 0: row r codes tok[r], pair r; mode 1: row r is position r % W of window first_win + r / W,
// its pair goes to element pair_tile_index(window - pair_win0, position) of the window tiles.
// row_max: [rows] float_key of each row's maximum; have_max false: computed into it first
void launch_cdf_pairs(const float* logits, int64_t rows, int V, int P, const uint32_t* tab, const uint16_t* tok,
                      int64_t n_tok, int W, int64_t first_win, uint32_t* start,
                      uint32_t* freq, int mode, cudaStream_t s, int64_t pair_win0, uint32_t* row_max,
                      bool have_max);
void launch_quantize_cdf(const float* logits, int64_t rows, int V, int P, const uint32_t* tab, uint32_t* cdf,
                         cudaStream_t s);
// launch_cdf_pairs over the restricted alphabet (no row_max input); a token outside it sets
// kErrCorrupt in *err and gets the pair (0, 1)
void launch_cdf_pairs_alpha(const float* logits, int64_t rows, int V, int P, const uint32_t* tab,
                            const uint16_t* tok, int64_t n_tok, int W, int64_t first_win, uint32_t* start, uint32_t* freq, int mode, cudaStream_t s, int64_t pair_win0,
                            const AlphaIds& alpha, uint32_t* err);
void launch_dec_search_alpha(const float* logits, int64_t n, int V, int P, const uint32_t* tab, void* dec_state,
                             const uint8_t* codes, uint16_t* sym_out, int64_t sym_stride, int64_t pos,
                             const uint32_t* win_len, const AlphaIds& alpha, uint32_t* err, cudaStream_t s);
void launch_dec_search(const float* logits, int64_t n, int V, int P, const uint32_t* tab, void* dec_state,
                       const uint8_t* codes, uint16_t* sym_out, int64_t sym_stride, int64_t pos,
                       const uint32_t* win_len, uint32_t* err, cudaStream_t s);

// coder.cu
// Window tiles: the coder's input layout on the encode path. The (start, freq) pairs of 32
// consecutive windows and 8 consecutive positions form one tile of 256 elements, element
// (w % 32) * 8 + i % 8; tiles follow each other by window block, then by position group, with
// G = ceil(W / 8) groups per window. A thread reading its window's 8 tokens of a group reads two
// 16-byte vectors, and a warp's 32 threads one contiguous kilobyte per array.
__host__ __device__ __forceinline__ int64_t pair_tile_groups(int64_t W) { return (W + 7) >> 3; }
__host__ __device__ __forceinline__ int64_t pair_tile_index(int64_t w, int64_t i, int64_t groups) {
  return (((w >> 5) * groups + (i >> 3)) << 8) + ((w & 31) << 3) + (i & 7);
}
// elements of a tiled pair array for n_win windows of W positions (whole tiles)
__host__ __device__ __forceinline__ int64_t pair_tile_elems(int64_t n_win, int64_t W) {
  return ((n_win + 31) >> 5) * pair_tile_groups(W) * 256;
}
size_t slot_bytes(size_t win_tokens, int P);
// pairs at start[w * stride_win + i * stride_pos] (tiled = false) or in window tiles (tiled =
// true, strides ignored); check: validate every pair (entry points taking a caller's pairs)
void launch_range_encode(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                         const uint32_t* win_len, int64_t stride_win, int64_t stride_pos, uint8_t* slots,
                         size_t slot_sz, uint32_t* bitlen, uint32_t* err, cudaStream_t s, bool tiled = false,
                         bool check = true);
// interleaved: the slots as the tiled coder leaves them, each 32-window block one table whose
// 16-byte chunk c of window w lies at ((c * 32 + w % 32) * 16) from the block's first slot
void launch_pack_codes(const uint8_t* slots, size_t slot_sz, const uint32_t* bitlen, int64_t n_win,
                       uint64_t* offsets /* [n_win+1] scratch */, uint8_t* out, cudaStream_t s, bool interleaved);
// crc32 of the little-endian bytes of tok[w * stride .. w * stride + len[w]) for each w < n_win
void launch_window_crc(const uint16_t* tok, int64_t stride, const uint32_t* len, int64_t n_win, uint32_t* out,
                       cudaStream_t s);
size_t dec_state_bytes();
void launch_dec_init(const uint8_t* codes, const uint64_t* code_off, const uint32_t* bitlen, int64_t n,
                     void* state, cudaStream_t s);

// attn_tc.cu (tcgen05). q: [q_rows][q_dim] (query head h at column h * hd); kv: [kv_rows][kv_dim]
// (key head j at column k_off + j * hd, value head j at v_off + j * hd)
bool tc_attention_supported(int hd, int64_t qkv_dim);
void launch_attention_tc(const void* q, int64_t q_rows, int64_t q_dim, const void* kv, int64_t kv_rows,
                         int64_t kv_dim, int k_off, int v_off, void* out, int64_t out_stride, int nq, int nkv, int hd,
                         int W, int64_t n_win,
                         int64_t pos_first, int n_pos, int64_t q_win_stride, uint32_t* err, cudaStream_t s);

// gemm_tc.cu (tcgen05)
bool tc_gemm_supported(int64_t M, int64_t N, int64_t K, int epi = 0);
void launch_gemm_tc(const void* A, const void* B, void* C, int64_t M, int64_t N, int64_t K, int epi, uint32_t* err,
                    cudaStream_t s, const RopeArgs* rope = nullptr, const NormArgs* norm = nullptr);
// x[r][:] = E[tok_in[r]][:] (fp32), xh = fp16(x), ss[r * (d/256) + k] = sum of squares of columns
// [256k, 256k + 256) of row r (d % 256 == 0)
void launch_embed_fused(const uint16_t* tok_in, int64_t rows, const void* E, int d, float* x, __half* xh, float* ss,
                        cudaStream_t s);

}  // namespace lmgc
