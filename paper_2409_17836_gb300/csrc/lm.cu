// lm.cu -- the LM prior of Eq. 2 (a Llama-family decoder, Sec. 5.1): weight generation,
// embedding, RMSNorm, RoPE, SwiGLU (the kernels bf16 models do not fold into their GEMM
// epilogues, and fp32 models use). The dense contractions and attention are on the tensor cores
// (gemm_tc.cu, attn_tc.cu; gemm_tf32.cu, attn_tf32.cu for fp32 models).
//
// Every kernel here is row-invariant: a row's result depends only on that row's inputs (and, for
// attention, on the keys/values of its window), never on M, the batch or the row's place in a
// tile. That is what lets the decoder (one row per window per step) reproduce the encoder's
// logits bit for bit.
#include <math.h>

#include <algorithm>

#include "lmgc_internal.cuh"

namespace lmgc {

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__half>(__half v) { return __half2float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __half from_f<__half>(float v) { return __float2half_rn(v); }

// ------------------------------------------------------------------------------------------
// Random-init weights: splitmix64 (Steele, Lea, Flood 2014) of seed ^ (tensor_id << 40) ^ index;
// top 24 bits u; w = fp32((u - 2^23) * 2^-23) * a, a = fp32(init_std * sqrt(3)).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// A bf16 model keeps its bf16-valued weights in fp16 containers (every bf16 value with magnitude
// >= 2^-17 is exact in fp16; smaller ones round to the 2^-24 grid of fp16 subnormals).
template <typename T>
constexpr bool kBf16Values = false;
template <>
constexpr bool kBf16Values<__half> = true;

template <typename T>
__global__ void k_init_weights(T* __restrict__ dst, uint64_t seed, uint32_t tid, int64_t rows, int64_t cols,
                               int64_t ld, int64_t row_off, int64_t rblk, int64_t rstride, float a) {
  const int64_t total = rows * cols;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    uint64_t u = splitmix64(seed ^ ((uint64_t)tid << 40) ^ (uint64_t)idx) >> 40;
    float unit = (float)((int32_t)u - (1 << 23)) * (1.0f / 8388608.0f);
    float w = __fmul_rn(unit, a);
    if (kBf16Values<T>) w = __bfloat162float(__float2bfloat16_rn(w));  // the bf16 model's weight value
    int64_t r = idx / cols, c = idx - r * cols;
    const int64_t dr = row_off + (r / rblk) * rstride + r % rblk;
    dst[dr * ld + c] = from_f<T>(w);
  }
}

void launch_init_weights(void* dst, int dtype, uint64_t seed, uint32_t tid, int64_t rows, int64_t cols, int64_t ld,
                         int64_t row_off, float init_std, cudaStream_t s, int64_t rblk, int64_t rstride) {
  if (rblk <= 0) {
    rblk = rows;
    rstride = 0;
  }
  float a = (float)((double)init_std * sqrt(3.0));
  int64_t total = rows * cols;
  unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 152 * 64);
  note_launch();
  if (dtype == LMGC_BF16)
    k_init_weights<<<blocks, 256, 0, s>>>((__half*)dst, seed, tid, rows, cols, ld, row_off, rblk, rstride, a);
  else
    k_init_weights<<<blocks, 256, 0, s>>>((float*)dst, seed, tid, rows, cols, ld, row_off, rblk, rstride, a);
}

// ------------------------------------------------------------------------------------------
// Window inputs (Eq. 2): window w's model input is [BOS, t_{wW}, ..., t_{wW+W-2}]; positions past
// the end of the token stream read padding id 0.
// ------------------------------------------------------------------------------------------
__global__ void k_window_inputs(const uint16_t* __restrict__ tok, int64_t n_tok, int64_t first_win, int64_t n_win,
                                int W, uint16_t* __restrict__ tok_in) {
  int64_t total = n_win * W;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < total; r += (int64_t)gridDim.x * blockDim.x) {
    int64_t wl = r / W;
    int i = (int)(r - wl * W);
    int64_t g = (first_win + wl) * W + i - 1;
    tok_in[r] = i == 0 ? (uint16_t)kTokBos : (g < n_tok ? tok[g] : (uint16_t)0);
  }
}

void launch_window_inputs(const uint16_t* tok, int64_t n_tok, int64_t first_win, int64_t n_win, int W,
                          uint16_t* tok_in, cudaStream_t s) {
  int64_t total = n_win * W;
  unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 152 * 32);
  note_launch();
  k_window_inputs<<<blocks, 256, 0, s>>>(tok, n_tok, first_win, n_win, W, tok_in);
}

// x[r][:] = E[tok_in[r]][:] (fp32 residual stream)
template <typename T>
__global__ void k_embed(const uint16_t* __restrict__ tok_in, int64_t rows, const T* __restrict__ E, int d,
                        float* __restrict__ x) {
  int64_t r = blockIdx.x;
  if (r >= rows) return;
  const T* e = E + (int64_t)tok_in[r] * d;
  for (int j = threadIdx.x; j < d; j += blockDim.x) x[r * d + j] = to_f<T>(e[j]);
}

void launch_embed(const uint16_t* tok_in, int64_t rows, const void* E, int d, int dtype, float* x, cudaStream_t s) {
  if (rows <= 0) return;
  note_launch();
  if (dtype == LMGC_BF16) k_embed<<<(unsigned)rows, 128, 0, s>>>(tok_in, rows, (const __half*)E, d, x);
  else k_embed<<<(unsigned)rows, 128, 0, s>>>(tok_in, rows, (const float*)E, d, x);
}

// Embedding for the fused-RMSNorm path: 8 warps per row; warp w handles the 256-column chunks
// w, w + 8, ...; each chunk's sum of squares is reduced in a fixed order.
__global__ void __launch_bounds__(256) k_embed_fused(const uint16_t* __restrict__ tok_in, int64_t rows,
                                                     const __half* __restrict__ E, int d, float* __restrict__ x,
                                                     __half* __restrict__ xh, float* __restrict__ ss) {
  const int64_t r = blockIdx.x;
  if (r >= rows) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const __half* e = E + (int64_t)tok_in[r] * d;
  const int parts = d / 256;
  for (int k = warp; k < parts; k += 8) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 8; i++) {
      const int c = k * 256 + i * 32 + lane;
      const __half hv = e[c];
      const float v = __half2float(hv);
      x[r * d + c] = v;
      xh[r * d + c] = hv;
      acc += v * v;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) ss[r * parts + k] = acc;
  }
}

void launch_embed_fused(const uint16_t* tok_in, int64_t rows, const void* E, int d, float* x, __half* xh, float* ss,
                        cudaStream_t s) {
  if (rows <= 0) return;
  note_launch();
  k_embed_fused<<<(unsigned)rows, 256, 0, s>>>(tok_in, rows, (const __half*)E, d, x, xh, ss);
}

// ------------------------------------------------------------------------------------------
// RMSNorm with unit gain: y = x * rsqrt(mean(x^2) + eps). One warp per row; a fixed reduction
// order (per-lane sequential, then a butterfly) keeps it row-invariant.
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_rmsnorm(const float* __restrict__ x, int64_t rows, int d, float eps,
                                                 T* __restrict__ y) {
  int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float4* xr = reinterpret_cast<const float4*>(x + r * d);
  float ss = 0.f;
  for (int j = lane; j < d / 4; j += 32) {
    float4 v = xr[j];
    ss += v.x * v.x;
    ss += v.y * v.y;
    ss += v.z * v.z;
    ss += v.w * v.w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  float inv = rsqrtf(ss / (float)d + eps);
  T* yr = y + r * d;
  for (int j = lane; j < d / 4; j += 32) {
    float4 v = xr[j];
    yr[4 * j + 0] = from_f<T>(v.x * inv);
    yr[4 * j + 1] = from_f<T>(v.y * inv);
    yr[4 * j + 2] = from_f<T>(v.z * inv);
    yr[4 * j + 3] = from_f<T>(v.w * inv);
  }
}

void launch_rmsnorm(const float* x, int64_t rows, int d, float eps, void* out, int dtype, cudaStream_t s) {
  if (rows <= 0) return;
  note_launch();
  unsigned blocks = (unsigned)((rows + 7) / 8);
  if (dtype == LMGC_BF16) k_rmsnorm<<<blocks, 256, 0, s>>>(x, rows, d, eps, (__half*)out);
  else k_rmsnorm<<<blocks, 256, 0, s>>>(x, rows, d, eps, (float*)out);
}

// ------------------------------------------------------------------------------------------
// RoPE, rotate-half pairing: in each head, dims i and i + hd/2 rotate by pos * theta^(-2i/hd).
// Applied in place to the first n_rot_heads heads of each qkv row (the q heads then the k heads).
// Row r sits at position pos_first + (r mod q_win_stride).
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void k_rope(T* __restrict__ qkv, int64_t rows, int qkv_dim, int n_rot_heads, int hd,
                       const float2* __restrict__ cs, int64_t pos_first, int64_t q_win_stride) {
  const int half = hd / 2;
  const int64_t per_row = (int64_t)n_rot_heads * half;
  const int64_t total = rows * per_row;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    int64_t r = e / per_row;
    int rem = (int)(e - r * per_row);
    int h = rem / half, i = rem - h * half;
    int64_t pos = pos_first + (r % q_win_stride);
    float2 c = cs[pos * half + i];
    T* v = qkv + r * qkv_dim + (int64_t)h * hd;
    float a = to_f<T>(v[i]), b = to_f<T>(v[i + half]);
    v[i] = from_f<T>(a * c.x - b * c.y);
    v[i + half] = from_f<T>(a * c.y + b * c.x);
  }
}

void launch_rope(void* qkv, int64_t rows, int qkv_dim, int n_rot_heads, int hd, const float2* cs, int W,
                 int64_t pos_first, int64_t q_win_stride, int n_pos, int dtype, cudaStream_t s) {
  (void)W;
  (void)n_pos;
  int64_t total = rows * n_rot_heads * (hd / 2);
  if (total <= 0) return;
  note_launch();
  unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 152 * 32);
  if (dtype == LMGC_BF16)
    k_rope<<<blocks, 256, 0, s>>>((__half*)qkv, rows, qkv_dim, n_rot_heads, hd, cs, pos_first, q_win_stride);
  else k_rope<<<blocks, 256, 0, s>>>((float*)qkv, rows, qkv_dim, n_rot_heads, hd, cs, pos_first, q_win_stride);
}

// act[r][j] = silu(g) * u, g = gu[r][j], u = gu[r][ffn + j]
template <typename T>
__global__ void k_swiglu(const T* __restrict__ gu, int64_t rows, int ffn, T* __restrict__ act) {
  int64_t total = rows * ffn;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    int64_t r = e / ffn;
    int j = (int)(e - r * ffn);
    float g = to_f<T>(gu[r * 2 * ffn + j]);
    float u = to_f<T>(gu[r * 2 * ffn + ffn + j]);
    act[e] = from_f<T>(g / (1.f + expf(-g)) * u);
  }
}

void launch_swiglu(const void* gu, int64_t rows, int ffn, void* act, int dtype, cudaStream_t s) {
  int64_t total = rows * ffn;
  if (total <= 0) return;
  note_launch();
  unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 152 * 32);
  if (dtype == LMGC_BF16) k_swiglu<<<blocks, 256, 0, s>>>((const __half*)gu, rows, ffn, (__half*)act);
  else k_swiglu<<<blocks, 256, 0, s>>>((const float*)gu, rows, ffn, (float*)act);
}

// dst[(w * dst_win_stride + dst_pos) * row_elems + c] = src[w * src_stride + c]
template <typename T>
__global__ void k_copy_rows(const T* __restrict__ src, int64_t src_stride, T* __restrict__ dst, int64_t dst_win_stride,
                            int64_t dst_pos, int64_t n_rows, int64_t row_elems) {
  int64_t total = n_rows * row_elems;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    int64_t w = e / row_elems, c = e - w * row_elems;
    dst[(w * dst_win_stride + dst_pos) * row_elems + c] = src[w * src_stride + c];
  }
}

void launch_copy_rows(const void* src, int64_t src_stride, void* dst, int64_t dst_win_stride, int64_t dst_pos,
                      int64_t n_rows, int64_t row_elems, int dtype, cudaStream_t s) {
  int64_t total = n_rows * row_elems;
  if (total <= 0) return;
  note_launch();
  unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 152 * 32);
  if (dtype == LMGC_BF16)
    k_copy_rows<<<blocks, 256, 0, s>>>((const __half*)src, src_stride, (__half*)dst, dst_win_stride,
                                       dst_pos, n_rows, row_elems);
  else
    k_copy_rows<<<blocks, 256, 0, s>>>((const float*)src, src_stride, (float*)dst, dst_win_stride, dst_pos, n_rows,
                                       row_elems);
}

}  // namespace lmgc
