/*
 * lmgc.h -- C ABI of liblmgc.so, the GB300 (sm_103a) encode path of LM-GC
 * ("Language Models as Zero-shot Lossless Gradient Compressors", arXiv 2409.17836).
 *
 * The method (Sec. 4): serialise fp32 gradients into hex-digit text with separators, feed it in
 * fixed windows, each starting from BOS, to a causal language model whose next-token
 * distributions (Eq. 2) drive an arithmetic coder (Sec. 3). Decoding runs the model token by token
 * from BOS until the window is full (Sec. 4 "Compression").
 *
 * Conventions for every call:
 *  - Pointers named d_* are DEVICE pointers owned by the caller (allocated on the device the
 *    context was created on); pointers named h_* are HOST pointers owned by the caller. The
 *    library owns the context, the model weights and its workspace.
 *  - Calls are stream-ordered on `stream` (a cudaStream_t; NULL = the legacy default stream).
 *    Outputs written through host pointers (sizes, counts) are valid when the call returns; such
 *    calls synchronise the stream internally. Device outputs are valid once the stream reaches
 *    the call's end.
 *  - A context is not reentrant: one call at a time per context.
 *  - Every call returns an lmgc_status. On error nothing is guaranteed about device outputs;
 *    lmgc_last_error() gives a message. LMGC_ERR_NO_SPACE writes the required size through the
 *    size pointer and no output.
 *  - Results are deterministic: the same input and configuration give the same bytes.
 *
 * Token alphabet (character-level reading of Sec. 4 / Fig. 1): hex digit v -> id v (0..15),
 * ' ' -> 16, ',' -> 17, ';' -> 18, BOS -> 19. The model's vocabulary has `vocab` >= 20 ids; the
 * coder codes over all of them (Eq. 2 is a distribution over the whole vocabulary), or, with
 * lmgc_config.alphabet = 1, over the ids the serialisation can emit only.
 */
#ifndef LMGC_H
#define LMGC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct lmgc_ctx lmgc_ctx;
typedef struct CUstream_st* lmgc_stream; /* the same type as cudaStream_t */

typedef enum {
  LMGC_OK = 0,
  LMGC_ERR_INVALID = -1,  /* bad argument or configuration */
  LMGC_ERR_NO_SPACE = -2, /* output capacity too small; required size written back */
  LMGC_ERR_CUDA = -3,     /* a CUDA runtime call failed */
  LMGC_ERR_CORRUPT = -4,  /* malformed container or code */
  LMGC_ERR_LIMIT = -5,    /* a device loop hit its iteration cap (reported, never spun) */
  LMGC_ERR_NOMEM = -6     /* device allocation failed */
} lmgc_status;

enum { LMGC_F32 = 0, LMGC_BF16 = 1 };

/* Separator modes (Table 1 serialisations): H_s, H_c, H_{c+s}, H_semi, H_n. */
enum { LMGC_SEP_SPACE = 0, LMGC_SEP_COMMA = 1, LMGC_SEP_COMMA_SPACE = 2, LMGC_SEP_SEMI = 3, LMGC_SEP_NONE = 4 };

/* Input kinds: fp32 gradient values (8 hex digits each, Sec. 4) or uint8 codes of the
 * lossy-compatible setting (Sec. 5.4, Eq. 4; 2 hex digits each). */
enum { LMGC_IN_F32 = 0, LMGC_IN_U8 = 1 };

/* Model and coder configuration. The model is a Llama-family decoder (the paper's LLMs,
 * Sec. 5.1): token embedding; per layer x += Wo Attn(RoPE(Wq n), RoPE(Wk n), Wv n) with
 * n = RMSNorm(x) and x += Wdown (silu(Wgate n') * Wup n') with n' = RMSNorm(x); a final RMSNorm;
 * logits = Wvocab x. Grouped-query attention when n_kv_heads < n_heads. Pretrained weights
 * are not available: every weight is drawn from splitmix64(weight_seed ^ (tensor_id << 40) ^
 * index), top 24 bits u, w = ((u - 2^23) * 2^-23) * fp32(init_std * sqrt(3)) (rounded to bf16
 * for dtype LMGC_BF16). */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, d_ffn, vocab;
  int32_t dtype;         /* LMGC_F32: fp32 weights and activations; LMGC_BF16: bf16-valued weights,
                            computed with fp16 activations and fp16 x fp16 -> fp32 MMAs (every bf16
                            value >= 2^-17 in magnitude is exact in fp16, smaller ones round to
                            the 2^-24 grid) */
  int32_t window;        /* W: tokens per independently coded window (Sec. 5.3 "Context window size") */
  int32_t cdf_bits;      /* P: the integer CDFs sum to 2^P; 2^P > vocab, P <= 30 */
  int32_t sep_mode;      /* LMGC_SEP_* */
  int32_t input_kind;    /* LMGC_IN_* */
  int32_t batch_windows; /* windows per model batch (workspace is sized for it) */
  uint64_t weight_seed;
  float init_std, rms_eps, rope_theta;
  int32_t byte_group;    /* bytes per separator group (Sec. 5.3 "Byte grouping", BPG 1..8); 0 = one
                            group per value (the default: BPG 4 for fp32, 1 for uint8 codes) */
  int32_t byte_order;    /* fp32 bytes in the stream: 0 most significant first, 1 least significant
                            first (uint8 codes: 0) */
  int32_t alphabet;      /* 0: each position's integer CDF spans the whole vocabulary (Sec. 4);
                            1: it spans only the ids the serialisation can emit (the 16 hex digits
                            and the separator ids of sep_mode), taken over those logits in
                            ascending id order, and a token is coded as its index among them. A
                            variant the paper does not describe. */
} lmgc_config;

/* Create a context on the current CUDA device: validates the configuration, allocates the
 * weights and the workspace for `batch_windows` windows and generates the weights on the device.
 * *out receives the context. Every contraction (the linear layers, attention, the vocabulary
 * projection) runs on the tcgen05 kernels, fp16 operands for LMGC_BF16 and three-pass TF32 for
 * LMGC_F32, with no other backend. Errors: INVALID (bad shape: d_model % n_heads,
 * n_heads % n_kv_heads, head dim not 64 or 128 for LMGC_BF16 or not 32 or 64 for LMGC_F32,
 * vocab < 20, cdf_bits out of range; a device or driver without the tcgen05 kernels and the
 * tensor-map encoder), NOMEM, CUDA. */
lmgc_status lmgc_create(const lmgc_config* cfg, lmgc_ctx** out);

/* Free everything the context owns. NULL is accepted. */
lmgc_status lmgc_destroy(lmgc_ctx* ctx);

/* Copy the last error message of ctx (or, for ctx == NULL, of the last failed call on this host
 * thread) into buf (NUL-terminated, truncated to len). */
lmgc_status lmgc_last_error(const lmgc_ctx* ctx, char* buf, size_t len);

/* Tokens per serialised value for the context's input kind and separator mode. Errors: INVALID
 * when byte groups cross values (byte_group 3, or 8 for fp32), so that no per-value count exists;
 * lmgc_serial_tokens gives the count of any n then. */
lmgc_status lmgc_tokens_per_value(const lmgc_ctx* ctx, size_t* tpv);

/* Token count of n serialised values: 2 digits per byte plus the separator tokens of
 * ceil(bytes / group) groups. Errors: INVALID. */
lmgc_status lmgc_serial_tokens(const lmgc_ctx* ctx, size_t n, size_t* n_tok);

/* Sec. 4 "Serialization" and Fig. 1: every 4 bits of a value become one hex digit, most
 * significant first (sign and exponent first), then the separator tokens. With byte_group or
 * byte_order set (Sec. 5.3 "Byte grouping"): the values' bytes in order (fp32 bytes per
 * byte_order), two hex digits per byte, high nibble first, and the separator after every
 * byte_group bytes and after a final partial group.
 * d_in: n values (fp32 bit patterns or uint8 codes per the context's input kind).
 * d_tok: uint16 token ids (capacity cap_tok). *n_tok receives lmgc_serial_tokens(n) (host).
 * Errors: INVALID, NO_SPACE (cap_tok too small; *n_tok = required), CUDA. */
lmgc_status lmgc_serialize(lmgc_ctx* ctx, const void* d_in, size_t n, uint16_t* d_tok, size_t cap_tok,
                           size_t* n_tok, lmgc_stream stream);

/* Inverse of lmgc_serialize. d_out receives the n values with lmgc_serial_tokens(n) = n_tok
 * (capacity cap_values). Errors: CORRUPT if no n gives n_tok tokens or a token is out of place;
 * NO_SPACE. Syncs. */
lmgc_status lmgc_deserialize(lmgc_ctx* ctx, const uint16_t* d_tok, size_t n_tok, void* d_out, size_t cap_values,
                             size_t* n_values, lmgc_stream stream);

/* Eq. 2 over windows: for windows w = first_win .. first_win + n_win - 1 of the token stream
 * d_tok[0 .. n_tok) (window w = tokens [w*W, min((w+1)*W, n_tok))), the model input is
 * [BOS, t_{wW}, ..., t_{wW+W-2}] and position i's logits are those of p(t_{wW+i} | BOS, t_<).
 * d_logits: fp32 [n_win][W][vocab] row-major. Rows past the end of a partial last window are
 * computed on padding input and must be ignored. n_win may exceed batch_windows (processed in
 * batches). Errors: INVALID (window range beyond the stream), CUDA. */
lmgc_status lmgc_lm_probs(lmgc_ctx* ctx, const uint16_t* d_tok, size_t n_tok, size_t first_win, size_t n_win,
                          float* d_logits, lmgc_stream stream);

/* The model's dense contraction (every linear layer of the Eq. 2 model and its vocabulary
 * projection), exposed for parity tests of the GEMM kernels: C[M][N] (op)= A[M][K] . B[N][K]^T,
 * A, B and C row-major and 16-byte aligned (bf16-weight contexts: fp16 on the tcgen05 kernel; fp32
 * contexts: fp32 on the tcgen05 kernel in three-pass TF32 form, each operand split into a TF32
 * high part and the remainder), fp32 accumulation in k order (for LMGC_BF16 contexts A and B are
 * fp16, see lmgc_config.dtype).
 * epi 0: C = result in the operand type; 1: fp32 C += result;
 * 2: fp32 C = result; 3 (bf16, N % 256 == 0): the SwiGLU MLP input -- B's rows hold gate and up
 * rows interleaved in 128-row blocks (rows 256t..256t+127 gate, 256t+128..256t+255 up) and
 * C[M][N/2] (fp16) = silu(gate) * up, i.e. C[m][128t+j] = silu(R[m][256t+j]) * R[m][256t+128+j];
 * 5: as 1, through the tensor-core kernel's 8-warp epilogue (the O projection's form).
 * Errors: INVALID (K % 8 != 0, A, B or C not 16-byte aligned, epi outside 0..3 and 5, epi 3
 * unsupported), LIMIT, CUDA. Syncs. */
lmgc_status lmgc_gemm(lmgc_ctx* ctx, const void* d_a, const void* d_b, void* d_c, size_t M, size_t N, size_t K,
                      int epi, lmgc_stream stream);

/* Integer CDF of each logit row (the coder input; the paper adapts Torchac, whose CDFs are
 * integers, Sec. 5.1). For a row z[0..V) with T = 2^P: m = max z; y_j = fp32(fp32(z_j - m) *
 * fp32(2^16 log2 e)); a_j = -rint(y_j) clamped to 40*2^16; e_j = 2^31 * 2^(-a_j/65536) in fixed
 * point from two 256-entry tables; g_j = floor(e_j (T - V) / sum e); freq_j = 1 + g_j with the
 * remainder added to the lowest-index largest e_j; cdf[0] = 0, cdf[V] = T. Rows always span the
 * whole vocabulary: the restricted alphabet (lmgc_config.alphabet) does not apply here; its CDF
 * is this one applied to the row's alphabet columns.
 * d_logits: fp32 [rows][V]; d_cdf: uint32 [rows][V+1]. Errors: INVALID, CUDA. */
lmgc_status lmgc_quantize_cdf(lmgc_ctx* ctx, const float* d_logits, size_t rows, uint32_t* d_cdf,
                              lmgc_stream stream);

/* The coder's per-token input without materialising CDFs: for row r with symbol d_sym[r],
 * d_start[r] = cdf_r[sym] and d_freq[r] = cdf_r[sym + 1] - cdf_r[sym] under the quantiser of
 * lmgc_quantize_cdf. All arrays are indexed by row. It runs the encode path's kernel, after a
 * pass that takes each row's maximum into stream-ordered scratch of 4 bytes per row (allocated
 * and freed on the stream). With alphabet 1 the quantiser runs over the restricted alphabet's
 * logits of each row (V' ids), sym is the index of d_sym[r] among them, and the call syncs to
 * report a d_sym[r] outside the alphabet (CORRUPT; its pair is (0, 1)).
 * Errors: INVALID, CORRUPT, CUDA (including a failed scratch allocation). */
lmgc_status lmgc_cdf_pairs(lmgc_ctx* ctx, const float* d_logits, size_t rows, const uint16_t* d_sym,
                           uint32_t* d_start, uint32_t* d_freq, lmgc_stream stream);

/* Arithmetic coder (Sec. 3 "Arithmetic coding"), one independent stream per window, in an exact
 * integer form: R = 2^62, L = 0, B = 0; per token r = R >> P, L += r*start, R = r*freq,
 * k = max(0, 62 - bitlen(R)), R <<= k, L <<= k, B += k; the code is the top B + 2 bits of
 * ceil(L / 2^60) * 2^60, most significant bit first, padded with zeros to a byte.
 * Token i of window w is read at d_start[w*stride_win + i*stride_pos] (same for d_freq; every
 * pair is checked: 0 < freq, start + freq <= 2^cdf_bits);
 * window w has d_win_len[w] tokens (device array), or win_tokens tokens when d_win_len is NULL.
 * d_out receives the codes of windows 0..n_win-1 back to back, each starting on a byte;
 * d_bitlen[w] (device) receives each code's bit length; *out_bytes (host) the total bytes.
 * Scratch: allocates stream-ordered device memory for one code slot per window.
 * Errors: INVALID (cdf_bits outside 1..30, a window longer than win_tokens), NO_SPACE
 * (cap < total; *out_bytes = required; d_bitlen is still written), CUDA. Syncs. */
lmgc_status lmgc_range_encode(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                              size_t win_tokens, const uint32_t* d_win_len, size_t stride_win, size_t stride_pos,
                              uint8_t* d_out, size_t cap, size_t* out_bytes, uint32_t* d_bitlen,
                              lmgc_stream stream);

/* lmgc_range_encode with the pairs in window tiles, the layout the encode path hands its coder:
 * the pairs of 32 consecutive windows and 8 consecutive positions form one tile of 256 elements,
 * tiles ordered by window block and then by position group. With G = ceil(win_tokens / 8), token
 * i of window w is element ((w / 32) * G + i / 8) * 256 + (w % 32) * 8 + i % 8 of d_start (and of
 * d_freq), arrays of lmgc_pair_tile_elems(n_win, win_tokens) elements, 16-byte aligned (INVALID
 * otherwise; elements past a window's length or past n_win are read but not used). Each thread
 * codes one window; a warp stages its 32 windows' tiles through shared memory with asynchronous
 * 16-byte copies.
 * validate != 0: every pair is checked as in lmgc_range_encode. validate == 0: the caller vouches
 * that every pair satisfies 0 < freq < 2^cdf_bits and start + freq <= 2^cdf_bits (as the encode
 * path's own pairs from its CDF kernels do) and the check is skipped; pairs that break this give
 * unspecified codes and bit lengths (each at most its slot's size) but no access outside the
 * call's buffers; the encode path runs this form on its own pairs. Same arithmetic, output and
 * errors as lmgc_range_encode; its scratch holds one code slot per window for whole blocks of 32
 * windows (the codes of a block are interleaved in 16-byte chunks). Syncs. */
lmgc_status lmgc_range_encode_tiled(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                                    size_t win_tokens, const uint32_t* d_win_len, int validate, uint8_t* d_out,
                                    size_t cap, size_t* out_bytes, uint32_t* d_bitlen, lmgc_stream stream);

/* Elements of one window-tiled pair array for n_win windows of win_tokens positions
 * (ceil(n_win / 32) * ceil(win_tokens / 8) * 256). */
lmgc_status lmgc_pair_tile_elems(size_t n_win, size_t win_tokens, size_t* elems);

/* lmgc_range_encode for callers that cannot allocate device memory (for example a process whose
 * device memory is held entirely by another allocator, or a latency-critical path where
 * cudaMalloc / cudaFree, which may synchronise the device, are not allowed). The paper has no
 * counterpart: this is a deployment variant of the coder above, with the same arguments, output
 * and errors. It allocates nothing: its scratch (a 256-byte error word, the payload offsets and
 * one code slot of slot(win_tokens, cdf_bits) = ceil((win_tokens*cdf_bits + 2) / 32 + 1) * 4 bytes,
 * rounded up to 16, per window) lives in one fixed 64 MiB device array that every GPU loading the
 * library keeps until exit. Calls needing more than 64 MiB of scratch (about 10,900 windows of
 * 2048 tokens at cdf_bits 24) fail with INVALID and a message giving both sizes.
 * Windows of more than 2^29 / cdf_bits tokens are rejected the same way.
 * The first call on a device does the set-up: it looks up the array's device address (once per
 * device, with that device current); make that first call before any stream capture begins.
 * All calls share the array and it keeps the last call's contents: calls that overlap on the GPU
 * (other streams, other host threads) race on it and must be serialised by the caller. Every
 * call reads the total size back to the host and synchronises `stream` before it returns. */
lmgc_status lmgc_range_encode_noalloc(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits, size_t n_win,
                                      size_t win_tokens, const uint32_t* d_win_len, size_t stride_win,
                                      size_t stride_pos, uint8_t* d_out, size_t cap, size_t* out_bytes,
                                      uint32_t* d_bitlen, lmgc_stream stream);

/* Largest container lmgc_encode can produce for n input values (header + length and checksum
 * tables + the coder's worst case of cdf_bits bits per token + 2 bits per window). */
lmgc_status lmgc_encode_bound(const lmgc_ctx* ctx, size_t n, size_t* bytes);

/* The whole encode path (Sec. 4): serialise -> windows from BOS -> model logits -> integer CDF
 * pairs -> one code per window -> container. Container layout (little-endian):
 *   0 "LMGC" | 4 u32 version=2 | 8 u64 n_values | 16 u64 n_tok | 24 u32 window | 28 u32 cdf_bits |
 *   32 u32 input_kind | 36 u32 serialisation = sep_mode | byte_group << 8 | byte_order << 16 |
 *   alphabet << 24 | 40 u32 vocab | 44 u32 n_win | 48 u64 weight_seed |
 *   56 u32 crc32 of the model shape | 60 u32 crc32 of bytes [0, 60) |
 *   64 u32 bitlen[n_win] | u32 crc_tok[n_win] | codes, ceil(bitlen/8) bytes each, in window order.
 * crc_tok[w] is the CRC-32 (IEEE 802.3) of window w's token ids as little-endian u16 bytes (the
 * window's own length), which lmgc_decode checks on every window it restores.
 * d_in: n values; d_out: capacity cap bytes. *out_bytes (host) = container size.
 * Errors: INVALID (n == 0), NO_SPACE (*out_bytes = required), CUDA. Syncs. */
lmgc_status lmgc_encode(lmgc_ctx* ctx, const void* d_in, size_t n, uint8_t* d_out, size_t cap, size_t* out_bytes,
                        lmgc_stream stream);

/* The windows [first_win, first_win + n_win) of lmgc_encode's container, for encoding a stream
 * sharded over several GPUs (windows are independent, Sec. 4 "Compression"): all n values are
 * serialised, only the given windows are modelled and coded. d_payload receives their codes
 * byte-aligned in window order (the container's payload slice), d_bitlen and d_crc (device, n_win
 * each) their bit lengths and token checksums, *payload_bytes (host) the slice size. A container
 * is the header of lmgc_container_header, the bit lengths of all windows in order, their token
 * checksums in order, then all payload slices in order. Errors: INVALID (range outside the
 * stream, null table pointer), NO_SPACE (*payload_bytes = required), CUDA. Syncs. */
lmgc_status lmgc_encode_windows(lmgc_ctx* ctx, const void* d_in, size_t n, size_t first_win, size_t n_win,
                                uint8_t* d_payload, size_t cap, size_t* payload_bytes, uint32_t* d_bitlen,
                                uint32_t* d_crc, lmgc_stream stream);

/* The 64-byte container header (layout under lmgc_encode) for n input values, written to the
 * host buffer h_header. */
lmgc_status lmgc_container_header(const lmgc_ctx* ctx, size_t n, uint8_t* h_header);

/* lmgc_encode with HOST buffers: copies h_in to the device, encodes, copies the container back
 * to h_out. The device staging buffers are owned by the context and reused across calls. */
lmgc_status lmgc_encode_host(lmgc_ctx* ctx, const void* h_in, size_t n, uint8_t* h_out, size_t cap,
                             size_t* out_bytes, lmgc_stream stream);

/* The KV-cached autoregressive inverse (Sec. 4 "Compression": decoding starts from BOS and runs
 * until the window is full). Decodes the windows h_win_ids[0 .. n_ids) (host array) of the
 * container d_in (device, in_bytes) into d_tok (device, [n_ids][W] uint16; a partial last window
 * fills only its length). Each decode step runs the same kernels as lmgc_encode on one row per
 * window, so its logits -- and hence its CDFs -- are bit-identical to the encoder's. Windows
 * are decoded in batches of as many as a KV cache of half the free device memory holds (the
 * cache keeps each position's keys and values, 2 n_kv_heads hd values per layer); the context
 * keeps that cache for later calls (lmgc_destroy frees it).
 * Errors: CORRUPT (bad header, a model or serialisation word -- separators, byte grouping and
 * order, alphabet -- other than the context's, a code that leaves its interval, or a restored
 * window whose token checksum differs from the container's), INVALID
 * (window id out of range), NO_SPACE (cap_tok < n_ids * W), CUDA. Syncs. */
lmgc_status lmgc_decode(lmgc_ctx* ctx, const uint8_t* d_in, size_t in_bytes, const uint32_t* h_win_ids,
                        size_t n_ids, uint16_t* d_tok, size_t cap_tok, lmgc_stream stream);

/* The number of windows lmgc_decode would take per batch if called now: as many as a KV cache of
 * half the free device memory (or the cache the context already holds, if larger) takes, at most
 * batch_windows * W (one workspace row per window). A build choice with no counterpart in the
 * paper, for callers sizing their decode requests. Errors: INVALID (null argument), CUDA. */
lmgc_status lmgc_decode_batch_windows(lmgc_ctx* ctx, size_t* n);

/* Per-stage device time of the last lmgc_encode call, in milliseconds (CUDA events):
 * ms[0] serialise, ms[1] model forward (all layers and the vocabulary projection),
 * ms[2] CDF pairs, ms[3] coder, ms[4] container assembly. n_ms: capacity of ms. */
lmgc_status lmgc_stage_times(const lmgc_ctx* ctx, float* ms, size_t n_ms);

/* Number of kernels this library has launched in the process so far (all contexts). */
lmgc_status lmgc_launch_count(uint64_t* n);

/* Kernel-class timing for roofline reports. lmgc_profile(ctx, 1) clears the counters and starts
 * recording a CUDA event pair around every launch of the classes below on the launching stream;
 * lmgc_profile(ctx, 0) stops. lmgc_kernel_stats returns, for class cls, its name, the launches
 * and summed device milliseconds recorded, and the summed algorithmic work of those launches
 * (flops for 0 "gemm" and 1 "attention"; bytes for 2 "cdf_pairs", 3 "range_encode",
 * 4 "serialize"; 0 for 5 "norm_rope_act" and 6 "other"). ctx == NULL selects the process-wide
 * counters of the context-free entry points (lmgc_range_encode: its coder kernel, class 3).
 * Errors: INVALID (cls outside 0..6). */
lmgc_status lmgc_profile(lmgc_ctx* ctx, int enable);
lmgc_status lmgc_kernel_stats(const lmgc_ctx* ctx, int cls, char* name, size_t name_len, int* launches, float* ms,
                              double* work);

#ifdef __cplusplus
}
#endif
#endif /* LMGC_H */
