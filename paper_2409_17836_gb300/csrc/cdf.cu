// cdf.cu -- logits -> integer CDF -> (start, freq) of the coded token, plus the decoder's
// symbol search.
//
// The coder of Sec. 3 needs the model's distribution p(t | BOS, t_<) (Eq. 2) as an integer CDF
// (the paper adapts Torchac, whose CDFs are integers; Sec. 5.1). For a row z[0..V), T = 2^P:
//   m = max z; y_j = fp32(fp32(z_j - m) * C), C = fp32(2^16 log2 e); a_j = -rint(y_j) (<= 40*2^16)
//   e_j = ((H[(a>>8)&255] * L[a&255] + 2^30) >> 31) >> (a >> 16),   H[h] = round(2^31 2^(-h/256)),
//         L[l] = round(2^31 2^(-l/65536))  -- a fixed-point 2^31 * exp(z_j - m)
//   S = sum e_j; g_j = floor(e_j (T - V) / S); freq_j = 1 + g_j; the remainder (T - V) - sum g_j
//   goes to the lowest index of the largest e_j; cdf[j] = sum_{i<j} freq_i.
// Only the fp32 subtract/multiply and rint touch floating point; the rest is integer, so the
// result is bit-exact on any machine that rounds fp32 to nearest.
//
// The encode path never materialises a CDF (V = 32000 would be 128 KB per token): one block per
// row reduces max, sum e and argmax, then sum_{j<s} g_j and g_s for the row's symbol s.
// floor(e (T - V) / S) uses a 32-bit fixed-point reciprocal of S and one exact remainder test.
#include <math.h>

#include <algorithm>

#include "lmgc_internal.cuh"

namespace lmgc {

// Tables H and L, computed in binary64 (each entry is >= 1e-4 away from a rounding tie, which
// is checked, so binary64 rounding cannot change them).
void upload_exp2_tables(uint32_t* d_tab, cudaStream_t s) {
  static uint32_t tab[512];
  static bool built = false;
  if (!built) {
    for (int i = 0; i < 256; i++) {
      double h = ldexp(exp2(-(double)i / 256.0), 31);
      double l = ldexp(exp2(-(double)i / 65536.0), 31);
      double fh = h - floor(h), fl = l - floor(l);
      if (fabs(fh - 0.5) < 1e-4 || fabs(fl - 0.5) < 1e-4) {
        // cannot happen for these tables; refuse to guess
        tab[0] = 0;
        return;
      }
      tab[i] = (uint32_t)llround(h);
      tab[256 + i] = (uint32_t)llround(l);
    }
    built = true;
  }
  cudaMemcpyAsync(d_tab, tab, sizeof(tab), cudaMemcpyHostToDevice, s);
  cudaStreamSynchronize(s);
}

constexpr int kCdfThreads = 512;
constexpr int kAMax = 40 * 65536;

// a = -rint(fp32(fp32(z - m) * C)) capped at 40 * 2^16: 2^(-a / 2^16) approximates exp(z - m).
// a = 0 exactly where e reaches its maximum 2^31, so the row's lowest-index argmax of e is its
// lowest index with a = 0.
__device__ __forceinline__ int exp2_code(float z, float m) {
  const float C = (float)(65536.0 * 1.4426950408889634073599246810019);
  const float y = __fmul_rn(__fsub_rn(z, m), C);  // <= 0: m is the row maximum
  // rint (ties to even) after clamping y to -40 * 2^16 (an integer, so rint keeps it), taken by
  // adding 1.5 * 2^23 in round-to-nearest-even: the sum lies in [2^23, 2^24), where fp32 spacing
  // is 1, so its low mantissa bits are 2^22 + rint(y)
  const float t = __fadd_rn(fmaxf(y, -(float)kAMax), 12582912.f);
  return (int)(0x4B400000u - __float_as_uint(t));
}

__device__ __forceinline__ uint32_t exp2_from_code(int a, const uint32_t* __restrict__ H,
                                                   const uint32_t* __restrict__ L) {
  // H, L <= 2^31, so (H L + 2^30) >> 31 <= 2^31 fits 32 bits; the final shift by a >> 16 (<= 40)
  // uses shr.b32, which yields 0 for shifts of 32 or more
  const uint64_t hl = (uint64_t)H[(a >> 8) & 255] * (uint64_t)L[a & 255];
  const uint32_t e31 = (uint32_t)((hl + (1ull << 30)) >> 31);
  uint32_t e;
  asm("shr.b32 %0, %1, %2;" : "=r"(e) : "r"(e31), "r"(a >> 16));
  return e;
}

__device__ __forceinline__ uint32_t exp2_fixed(float z, float m, const uint32_t* __restrict__ H,
                                               const uint32_t* __restrict__ L) {
  return exp2_from_code(exp2_code(z, m), H, L);
}

template <typename V>
__device__ __forceinline__ V warp_sum(V v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide reductions (kCdfThreads threads). `red` is shared scratch of >= 32 entries.
__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  v = lane < (kCdfThreads / 32) ? red[lane] : -INFINITY;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ uint64_t block_sum_u64(uint64_t v, uint64_t* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  v = lane < (kCdfThreads / 32) ? red[lane] : 0ull;
  return warp_sum(v);
}

__device__ __forceinline__ int block_min_int(int v, int* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  v = lane < (kCdfThreads / 32) ? red[lane] : 0x7fffffff;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

struct RowStats {
  float m;
  uint64_t S, Mq;
  uint32_t F;  // floor(Mq * 2^32 / S): floor(e * Mq / S) is (e * F) >> 32 or one more
  int amax;
};

// g = floor(e * Mq / S) exactly: q0 = (e F) >> 32 satisfies g - 1 <= q0 <= g (e <= 2^31 and
// S >= 2^31, the largest e being 2^31), and q0 S <= e Mq < 2^61, so one remainder test fixes it.
__device__ __forceinline__ uint64_t gfloor(uint32_t e, const RowStats& st) {
  const uint64_t X = (uint64_t)e * st.Mq;
  uint64_t q = __umulhi(e, st.F);
  if (X - q * st.S >= st.S) q++;
  return q;
}

// Rows whose start is 16-byte aligned and whose length is a multiple of 4 are read as float4.
__device__ __forceinline__ bool row_vec4(const float* z, int V) {
  return (V & 3) == 0 && (reinterpret_cast<uintptr_t>(z) & 15) == 0;
}

// Passes 1 and 2 over a row: max, sum of e, lowest-index argmax of e. With mkey (the float_key
// of the row's maximum, from the vocabulary GEMM's epilogue) the max pass is skipped.
__device__ __forceinline__ RowStats row_stats(const float* __restrict__ z, int V, int P, const uint32_t* H,
                                              const uint32_t* L, float* redf, uint64_t* redu,
                                              const uint32_t* mkey = nullptr) {
  RowStats st;
  const bool vec = row_vec4(z, V);  // block-uniform
  const float4* z4 = reinterpret_cast<const float4*>(z);
  const int V4 = V >> 2;
  float m = -INFINITY;
  if (mkey) {
    m = __uint_as_float(key_float_bits(*mkey));
  } else if (vec) {
    for (int j = threadIdx.x; j < V4; j += kCdfThreads) {
      const float4 v = __ldg(z4 + j);
      m = fmaxf(m, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)));
    }
  } else {
    for (int j = threadIdx.x; j < V; j += kCdfThreads) m = fmaxf(m, __ldg(z + j));
  }
  if (!mkey) m = block_max(m, redf);
  uint64_t S = 0;
  int best_j = 0x7fffffff;  // a thread's indices increase, so its first a = 0 is its lowest
  if (vec) {
    for (int j = threadIdx.x; j < V4; j += kCdfThreads) {
      const float4 v = __ldg(z4 + j);
      const int a0 = exp2_code(v.x, m), a1 = exp2_code(v.y, m), a2 = exp2_code(v.z, m), a3 = exp2_code(v.w, m);
      S += (uint64_t)exp2_from_code(a0, H, L) + (uint64_t)exp2_from_code(a1, H, L) +
           (uint64_t)exp2_from_code(a2, H, L) + (uint64_t)exp2_from_code(a3, H, L);
      if (min(min(a0, a1), min(a2, a3)) == 0 && best_j == 0x7fffffff)
        best_j = 4 * j + (a0 == 0 ? 0 : a1 == 0 ? 1 : a2 == 0 ? 2 : 3);
    }
  } else {
    for (int j = threadIdx.x; j < V; j += kCdfThreads) {
      const int a = exp2_code(__ldg(z + j), m);
      S += exp2_from_code(a, H, L);
      if (a == 0 && best_j == 0x7fffffff) best_j = j;
    }
  }
  S = block_sum_u64(S, redu);
  st.m = m;
  st.S = S;
  st.Mq = (1ull << P) - (uint64_t)V;
  st.F = (uint32_t)((st.Mq << 32) / S);
  st.amax = block_min_int(best_j, reinterpret_cast<int*>(redu));
  return st;
}

// sum of g = floor(e (T - V) / S) over the row (this thread's part)
__device__ __forceinline__ uint64_t row_gsum(const float* __restrict__ z, int V, const RowStats& st,
                                             const uint32_t* H, const uint32_t* L) {
  uint64_t gall = 0;
  if (row_vec4(z, V)) {
    const float4* z4 = reinterpret_cast<const float4*>(z);
    for (int j = threadIdx.x; j < (V >> 2); j += kCdfThreads) {
      const float4 v = __ldg(z4 + j);
      gall += gfloor(exp2_fixed(v.x, st.m, H, L), st) + gfloor(exp2_fixed(v.y, st.m, H, L), st) +
              gfloor(exp2_fixed(v.z, st.m, H, L), st) + gfloor(exp2_fixed(v.w, st.m, H, L), st);
    }
  } else {
    for (int j = threadIdx.x; j < V; j += kCdfThreads) gall += gfloor(exp2_fixed(__ldg(z + j), st.m, H, L), st);
  }
  return gall;
}

// ------------------------------------------------------------------------------------------
// Pairs of the coded tokens, one warp per row (the encode path). Per row the work is one read of
// the logits: the maximum comes with them (row_max: the float_key of each row's maximum, from the
// vocabulary GEMM's epilogue or from k_row_max_key), then one pass forms e_j and S = sum e_j. The
// symbol's start needs g_j = floor(e_j (T - V) / S) for j below the symbol only, plus the
// remainder (T - V) - sum g when the argmax of e (its lowest index with exponent code 0) lies
// below it, and its freq needs that remainder when the argmax is the symbol. So the pass over
// j <= sym also looks for code 0 there (the first one found is the argmax), and only then is the
// pass summing g over the whole row taken.
//
// Tables: H and L are held once per lane in shared memory, so a warp's 32 lookups fall in 32
// distinct banks whatever the indices (one wavefront each, against about three for one shared
// copy with random indices). Entry i of both tables sits at byte 256 i: lane c's copy of H2[i] at
// + 4c, of L[i] at + 128 + 4c, so each byte offset is one logic or byte-permute operation on a.
// H2[h] = 2 H[h] for h >= 1 and H2[0] = 2^32 - 1 (2 H[0] = 2^32 does not fit); then
// (H2 L + 2^31) >> 32 = (H L + 2^30) >> 31 for every (h, l) (for h = 0 because L <= 2^31), so
// the rounded product is the high word of one 32 x 32 + 64-bit multiply-add.
// The exponent code is not clamped: where the clamp would act (y < -40 * 2^16) the unclamped code
// is at least 40 * 2^16 as well, or (y < -2^22, -inf or NaN, where the rounding add leaves its
// exact range) at least 2^22 modulo 2^32, and e = 0 for both; a = 0 iff y rounds to 0 either way.
// Loads: 4 float4 per lane per stage and two stages in flight (the next stage is issued before
// the current one is reduced); the next row's first stage is issued before this row's epilogue.
// mode 0: row r codes d_sym[r]; pair index r.
// mode 1: rows are positions of windows first_win + r / W; the coded token is tok[w*W + i];
//         rows past the stream end are skipped; the pair goes to window w - pair_win0's element
//         of the coder's window tiles (pair_tile_index).
// ------------------------------------------------------------------------------------------
constexpr int kPairWarps = 16;
constexpr int kPairSmem = 256 * 256;  // 256 entries x (32 copies of H2, 32 copies of L), u32

// a = -rint(fp32(fp32(z - m) * C)) modulo 2^32 without the clamp (see above); mone = 2^32 - 1,
// passed at run time so that the subtraction is a multiply-add
__device__ __forceinline__ uint32_t exp2_code_u(float z, float m, uint32_t mone) {
  const float C = (float)(65536.0 * 1.4426950408889634073599246810019);
  const float t = __fadd_rn(__fmul_rn(__fsub_rn(z, m), C), 12582912.f);
  uint32_t a;
  asm("mad.lo.u32 %0, %1, %2, 0x4B400000;" : "=r"(a) : "r"(__float_as_uint(t)), "r"(mone));
  return a;
}

// e of exp2_from_code through this lane's table copies (tb: the tables' base; l4 = 4 lane,
// l4h = 4 lane + 128)
__device__ __forceinline__ uint32_t exp2_rep(uint32_t a, const char* tb, uint32_t l4, uint32_t l4h) {
  const uint32_t h2 = *reinterpret_cast<const uint32_t*>(tb + ((a & 0xFF00u) | l4));
  const uint32_t l = *reinterpret_cast<const uint32_t*>(tb + __byte_perm(a, l4h, 0x5504));
  const uint32_t e31 = (uint32_t)(((uint64_t)h2 * (uint64_t)l + 0x80000000ull) >> 32);
  uint32_t e;
  asm("shr.b32 %0, %1, %2;" : "=r"(e) : "r"(e31), "r"(a >> 16));
  return e;
}

// exp2_code_u of two logits at once: the subtraction and the multiply run as Blackwell's paired
// fp32 operations, which round each lane to nearest like __fsub_rn / __fmul_rn (z + (-m) equals
// z - m exactly, signed zeros included); the rounding add stays scalar. (With the add paired as
// well, the paired multiply and add came out singly rounded on GB300 -- codes off by one for a
// fraction of inputs -- while this form matched the scalar codes on every one of 3 million
// tested values.) nm2, c2 hold (-m, -m) and (C, C).
__device__ __forceinline__ void exp2_code_u2(float z0, float z1, uint64_t nm2, uint64_t c2, uint32_t mone,
                                             uint32_t& a0, uint32_t& a1) {
  uint64_t y;
  asm("{\n\t.reg .b64 d;\n\tmov.b64 d, {%1, %2};\n\tadd.rn.f32x2 d, d, %3;\n\tmul.rn.f32x2 %0, d, %4;\n\t}"
      : "=l"(y)
      : "f"(z0), "f"(z1), "l"(nm2), "l"(c2));
  float y0, y1;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(y0), "=f"(y1) : "l"(y));
  const uint32_t t0 = __float_as_uint(__fadd_rn(y0, 12582912.f)), t1 = __float_as_uint(__fadd_rn(y1, 12582912.f));
  asm("mad.lo.u32 %0, %1, %2, 0x4B400000;" : "=r"(a0) : "r"(t0), "r"(mone));
  asm("mad.lo.u32 %0, %1, %2, 0x4B400000;" : "=r"(a1) : "r"(t1), "r"(mone));
}

struct TabLane {
  const char* tb;
  uint32_t l4, l4h, one, mone;
  uint64_t nm2, c2;  // see exp2_code_u2
  __device__ __forceinline__ void set_max(float m) {
    const float C = (float)(65536.0 * 1.4426950408889634073599246810019);
    asm("mov.b64 %0, {%1, %1};" : "=l"(nm2) : "f"(-m));
    asm("mov.b64 %0, {%1, %1};" : "=l"(c2) : "f"(C));
  }
  __device__ __forceinline__ uint32_t code(float z, float m) const { return exp2_code_u(z, m, mone); }
  __device__ __forceinline__ uint32_t e(uint32_t a) const { return exp2_rep(a, tb, l4, l4h); }
  // S += e as one multiply-add by a 1 known only at run time
  __device__ __forceinline__ void acc(uint64_t& S, uint32_t x) const {
    asm("mad.wide.u32 %0, %1, %2, %0;" : "+l"(S) : "r"(x), "r"(one));
  }
  // four logits (set_max(m) done for this row)
  __device__ __forceinline__ void acc4(uint64_t& S, const float4& v) const {
    uint32_t a0, a1, a2, a3;
    exp2_code_u2(v.x, v.y, nm2, c2, mone, a0, a1);
    exp2_code_u2(v.z, v.w, nm2, c2, mone, a2, a3);
    acc(S, e(a0));
    acc(S, e(a1));
    acc(S, e(a2));
    acc(S, e(a3));
  }
  __device__ __forceinline__ uint64_t g4(const float4& v, float m, const RowStats& st) const {
    return gfloor(e(code(v.x, m)), st) + gfloor(e(code(v.y, m)), st) + gfloor(e(code(v.z, m)), st) +
           gfloor(e(code(v.w, m)), st);
  }
};

__device__ __forceinline__ float4 ld_stream4(const float4* p) {
  float4 v;
  asm("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];"
      : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
      : "l"(p));
  return v;
}

struct Stage4 {
  float4 v0, v1, v2, v3;
  __device__ __forceinline__ void load(const float4* p) {  // p: this lane's first float4 of the stage
    v0 = ld_stream4(p);
    v1 = ld_stream4(p + 32);
    v2 = ld_stream4(p + 64);
    v3 = ld_stream4(p + 96);
  }
  __device__ __forceinline__ void acc(uint64_t& S, const TabLane& t) const {
    t.acc4(S, v0);
    t.acc4(S, v1);
    t.acc4(S, v2);
    t.acc4(S, v3);
  }
};

__global__ void __launch_bounds__(32 * kPairWarps, 2) k_cdf_pairs(
    const float* __restrict__ logits, int64_t rows, int V, int P, const uint32_t* __restrict__ tab,
    const uint16_t* __restrict__ tok, int64_t n_tok, int W, int64_t first_win,
    uint32_t* __restrict__ start, uint32_t* __restrict__ freq, int mode, int64_t pair_win0,
    const uint32_t* __restrict__ row_max) {
  extern __shared__ __align__(16) uint32_t rep_tab[];  // [256][64]: H2 x 32, L x 32
  for (int i = threadIdx.x; i < 256 * 64; i += 32 * kPairWarps) {
    const int j = i >> 6;
    const uint32_t h = tab[j];
    rep_tab[i] = (i & 32) ? tab[256 + j] : (h >= 0x80000000u ? 0xFFFFFFFFu : 2u * h);
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  TabLane tl;
  tl.tb = reinterpret_cast<const char*>(rep_tab);
  tl.l4 = 4u * (uint32_t)lane;
  tl.l4h = tl.l4 | 128u;
  tl.one = (uint32_t)(P > 0);
  tl.mone = 0u - tl.one;
  const uint64_t Mq = (1ull << P) - (uint64_t)V;
  const int64_t step = (int64_t)gridDim.x * kPairWarps;
  // rows start 16-byte aligned and hold whole float4s (kernel-uniform)
  const bool vec = (V & 3) == 0 && (reinterpret_cast<uintptr_t>(logits) & 15) == 0;
  const int n4 = V >> 2;
  const int ng = vec ? n4 >> 7 : 0;  // whole stages of 128 float4s per row
  Stage4 A, B;
  int64_t r = (int64_t)blockIdx.x * kPairWarps + (threadIdx.x >> 5);
  if (r < rows && ng > 0) A.load(reinterpret_cast<const float4*>(logits + r * (int64_t)V) + lane);
  for (; r < rows; r += step) {
    const int64_t rn = r + step;
    const float4* zn = reinterpret_cast<const float4*>(logits + rn * (int64_t)V) + lane;
    int sym;
    int64_t out_idx;
    if (mode == 0) {
      sym = tok[r];
      out_idx = r;
    } else {
      const int64_t wl = r / W;
      const int i = (int)(r - wl * W);
      const int64_t gi = (first_win + wl) * W + i;
      if (gi >= n_tok) {  // warp-uniform; stage 0 of the next row replaces this row's
        if (rn < rows && ng > 0) A.load(zn);
        continue;
      }
      sym = tok[gi];
      out_idx = pair_tile_index(first_win + wl - pair_win0, i, pair_tile_groups(W));
    }
    const float* z = logits + r * (int64_t)V;
    const float4* z4 = reinterpret_cast<const float4*>(z) + lane;
    const float m = __uint_as_float(key_float_bits(row_max[r]));
    tl.set_max(m);
    uint64_t S = 0;
    if (vec) {
      int g = 0;
      for (; g + 2 <= ng; g += 2) {
        B.load(z4 + (g + 1) * 128);
        A.acc(S, tl);
        if (g + 2 < ng) A.load(z4 + (g + 2) * 128);
        B.acc(S, tl);
      }
      if (g < ng) A.acc(S, tl);
      if (rn < rows && ng > 0) A.load(zn);
      for (int j = ng * 128; j + lane < n4; j += 32) tl.acc4(S, ld_stream4(z4 + j));
    } else {
      for (int j = lane; j < V; j += 32) tl.acc(S, tl.e(tl.code(__ldg(z + j), m)));
    }
    RowStats st;
    st.m = m;
    st.S = warp_sum(S);
    st.Mq = Mq;
    st.F = st.S ? (uint32_t)((Mq << 32) / st.S) : 0u;  // S >= 2^31 when m is the row's maximum
    // g below the coded symbol and g of the symbol, packed as (below << 32) + at (each < 2^31),
    // and the lowest index <= sym with exponent code 0
    uint64_t packed = 0;
    int first0 = 0x7fffffff;
    for (int j = lane; j <= sym && j < V; j += 32) {
      const uint32_t a = tl.code(__ldg(z + j), m);
      const uint64_t g = gfloor(tl.e(a), st);
      packed += j < sym ? (g << 32) : g;
      if (a == 0u && first0 == 0x7fffffff) first0 = j;
    }
    packed = warp_sum(packed);
    const int amax = (int)__reduce_min_sync(0xffffffffu, (unsigned)first0);
    uint64_t gall = 0;
    if (amax <= sym) {  // warp-uniform: the argmax lies at or below the symbol
      if (vec) {
        for (int j = 0; j + lane < n4; j += 32) gall += tl.g4(__ldg(z4 + j), m, st);
      } else {
        for (int j = lane; j < V; j += 32) gall += gfloor(tl.e(tl.code(__ldg(z + j), m)), st);
      }
      gall = warp_sum(gall);
    }
    if (lane == 0) {
      const uint64_t resid = Mq - gall;
      start[out_idx] = (uint32_t)(sym + (packed >> 32) + (amax < sym ? resid : 0ull));
      freq[out_idx] = (uint32_t)(1ull + (packed & 0xFFFFFFFFull) + (amax == sym ? resid : 0ull));
    }
  }
}

// float_key of each row's maximum (one warp per row), for callers without the GEMM's maxima
__global__ void __launch_bounds__(256) k_row_max_key(const float* __restrict__ logits, int64_t rows, int V,
                                                     uint32_t* __restrict__ row_max) {
  const int lane = threadIdx.x & 31;
  const bool vec = (V & 3) == 0 && (reinterpret_cast<uintptr_t>(logits) & 15) == 0;
  for (int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5); r < rows; r += (int64_t)gridDim.x * 8) {
    const float* z = logits + r * (int64_t)V;
    uint32_t k = 0u;
    if (vec) {
      const float4* z4 = reinterpret_cast<const float4*>(z);
      for (int j = lane; j < (V >> 2); j += 32) {
        const float4 v = __ldg(z4 + j);
        k = max(max(k, max(float_key(__float_as_uint(v.x)), float_key(__float_as_uint(v.y)))),
                max(float_key(__float_as_uint(v.z)), float_key(__float_as_uint(v.w))));
      }
    } else {
      for (int j = lane; j < V; j += 32) k = max(k, float_key(__float_as_uint(__ldg(z + j))));
    }
    k = __reduce_max_sync(0xffffffffu, k);
    if (lane == 0) row_max[r] = k;
  }
}

void launch_cdf_pairs(const float* logits, int64_t rows, int V, int P, const uint32_t* tab, const uint16_t* tok,
                      int64_t n_tok, int W, int64_t first_win, uint32_t* start, uint32_t* freq, int mode,
                      cudaStream_t s, int64_t pair_win0, uint32_t* row_max, bool have_max) {
  if (rows <= 0) return;
  static int resident = 0;
  if (!resident) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaFuncSetAttribute(k_cdf_pairs, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_cdf_pairs, 32 * kPairWarps, kPairSmem);
    resident = std::max(1, sms * per_sm);
  }
  if (!have_max) {
    note_launch();
    k_row_max_key<<<(unsigned)std::min<int64_t>((rows + 7) / 8, 152 * 8), 256, 0, s>>>(logits, rows, V, row_max);
  }
  // one wave of resident blocks, each warp walking rows
  const int64_t blocks = std::min<int64_t>((rows + kPairWarps - 1) / kPairWarps, resident);
  note_launch();
  k_cdf_pairs<<<(unsigned)blocks, 32 * kPairWarps, kPairSmem, s>>>(logits, rows, V, P, tab, tok, n_tok, W,
                                                                   first_win, start, freq, mode, pair_win0, row_max);
}

// Block inclusive scan of one u64 per thread; returns the inclusive prefix; *total the tile sum.
__device__ __forceinline__ uint64_t block_scan_u64(uint64_t v, uint64_t* red, uint64_t* total) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint64_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) red[w] = x;
  __syncthreads();
  if (w == 0) {
    uint64_t y = lane < (kCdfThreads / 32) ? red[lane] : 0ull;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint64_t t = __shfl_up_sync(0xffffffffu, y, o);
      if (lane >= o) y += t;
    }
    if (lane < (kCdfThreads / 32)) red[lane] = y;
  }
  __syncthreads();
  uint64_t before = w > 0 ? red[w - 1] : 0ull;
  *total = red[kCdfThreads / 32 - 1];
  return x + before;
}

// Full CDF rows [rows][V+1] (parity and inspection).
__global__ void __launch_bounds__(kCdfThreads) k_quantize_cdf(const float* __restrict__ logits, int64_t rows, int V,
                                                              int P, const uint32_t* __restrict__ tab,
                                                              uint32_t* __restrict__ cdf) {
  __shared__ uint32_t H[256], L[256];
  __shared__ float redf[32];
  __shared__ uint64_t redu[32];
  __shared__ uint64_t scan_red[32];
  for (int i = threadIdx.x; i < 256; i += kCdfThreads) {
    H[i] = tab[i];
    L[i] = tab[256 + i];
  }
  __syncthreads();
  for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
    const float* z = logits + r * (int64_t)V;
    uint32_t* c = cdf + r * (int64_t)(V + 1);
    RowStats st = row_stats(z, V, P, H, L, redf, redu);
    const uint64_t gall = block_sum_u64(row_gsum(z, V, st, H, L), redu);
    const uint64_t resid = st.Mq - gall;
    uint64_t run = 0;
    if (threadIdx.x == 0) c[0] = 0;
    for (int j0 = 0; j0 < V; j0 += kCdfThreads) {
      int j = j0 + threadIdx.x;
      uint64_t f = 0;
      if (j < V) {
        f = 1 + gfloor(exp2_fixed(__ldg(z + j), st.m, H, L), st);
        if (j == st.amax) f += resid;
      }
      uint64_t tot;
      uint64_t inc = block_scan_u64(f, scan_red, &tot);
      if (j < V) c[j + 1] = (uint32_t)(run + inc);
      run += tot;
    }
  }
}

void launch_quantize_cdf(const float* logits, int64_t rows, int V, int P, const uint32_t* tab, uint32_t* cdf,
                         cudaStream_t s) {
  if (rows <= 0) return;
  unsigned blocks = (unsigned)std::min<int64_t>(rows, 152 * 4 * 8);
  note_launch();
  k_quantize_cdf<<<blocks, kCdfThreads, 0, s>>>(logits, rows, V, P, tab, cdf);
}

// ------------------------------------------------------------------------------------------
// Decoder step (Sec. 3: the decoder repeatedly looks up the interval holding the code value).
// State per window: R, D (62-bit window of the code value minus L), the code's bit position.
// t = D / (R >> P); the symbol s has cdf[s] <= t < cdf[s+1]; then D -= r cdf[s], R = r freq_s,
// k = 62 - bitlen(R), R <<= k, D = (D << k) | next k code bits.
// ------------------------------------------------------------------------------------------
struct DecState {
  uint64_t R, D;
  uint64_t bitpos;
  uint64_t code_off;
  uint64_t nbits;
};

size_t dec_state_bytes() { return sizeof(DecState); }

__device__ __forceinline__ uint32_t code_bit(const uint8_t* code, uint64_t nbits, uint64_t pos) {
  return pos < nbits ? (code[pos >> 3] >> (7 - (pos & 7))) & 1u : 0u;
}

__global__ void k_dec_init(const uint8_t* __restrict__ codes, const uint64_t* __restrict__ code_off,
                           const uint32_t* __restrict__ bitlen, int64_t n, DecState* __restrict__ st) {
  int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= n) return;
  DecState s;
  s.R = 1ull << 62;
  s.code_off = code_off[w];
  s.nbits = bitlen[w];
  s.D = 0;
  const uint8_t* code = codes + s.code_off;
  for (int i = 0; i < 62; i++) s.D = (s.D << 1) | code_bit(code, s.nbits, i);
  s.bitpos = 62;
  st[w] = s;
}

void launch_dec_init(const uint8_t* codes, const uint64_t* code_off, const uint32_t* bitlen, int64_t n, void* state,
                     cudaStream_t s) {
  if (n <= 0) return;
  note_launch();
  k_dec_init<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(codes, code_off, bitlen, n, (DecState*)state);
}

// One block per decoding window: quantise its logits row, find the symbol for the current code
// target, update the state. Windows whose length is <= pos are left unchanged.
__global__ void __launch_bounds__(kCdfThreads) k_dec_search(const float* __restrict__ logits, int64_t n, int V, int P,
                                                            const uint32_t* __restrict__ tab,
                                                            DecState* __restrict__ states,
                                                            const uint8_t* __restrict__ codes,
                                                            uint16_t* __restrict__ sym_out, int64_t sym_stride,
                                                            int64_t pos, const uint32_t* __restrict__ win_len,
                                                            uint32_t* err) {
  __shared__ uint32_t H[256], L[256];
  __shared__ float redf[32];
  __shared__ uint64_t redu[32];
  __shared__ uint64_t scan_red[32];
  __shared__ int found_s;
  __shared__ uint64_t found_lo, found_f;
  for (int i = threadIdx.x; i < 256; i += kCdfThreads) {
    H[i] = tab[i];
    L[i] = tab[256 + i];
  }
  __syncthreads();
  const int64_t w = blockIdx.x;
  if (w >= n || (int64_t)win_len[w] <= pos) return;
  DecState s = states[w];
  const uint64_t r = s.R >> P;
  const uint64_t t = s.D / r;
  const float* z = logits + w * (int64_t)V;
  RowStats st = row_stats(z, V, P, H, L, redf, redu);
  const uint64_t gall = block_sum_u64(row_gsum(z, V, st, H, L), redu);
  const uint64_t resid = st.Mq - gall;
  if (threadIdx.x == 0) found_s = -1;
  uint64_t run = 0;
  for (int j0 = 0; j0 < V; j0 += kCdfThreads) {
    int j = j0 + threadIdx.x;
    uint64_t f = 0;
    if (j < V) {
      f = 1 + gfloor(exp2_fixed(__ldg(z + j), st.m, H, L), st);
      if (j == st.amax) f += resid;
    }
    uint64_t tot;
    uint64_t inc = block_scan_u64(f, scan_red, &tot);
    uint64_t lo = run + inc - f;
    if (j < V && lo <= t && t < run + inc) {
      found_s = j;
      found_lo = lo;
      found_f = f;
    }
    run += tot;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  int sym = found_s;
  if (t >= (1ull << P) || sym < 0) {
    atomicOr(err, kErrCorrupt);
    sym = 0;
    found_lo = 0;
    found_f = 1;
  }
  s.D -= r * found_lo;
  s.R = r * found_f;
  int k = __clzll((long long)s.R) - 2;
  if (k < 0) k = 0;
  const uint8_t* code = codes + s.code_off;
  for (int i = 0; i < k; i++) s.D = (s.D << 1) | code_bit(code, s.nbits, s.bitpos + i);
  s.bitpos += k;
  s.R <<= k;
  states[w] = s;
  sym_out[w * sym_stride + pos] = (uint16_t)sym;
}

void launch_dec_search(const float* logits, int64_t n, int V, int P, const uint32_t* tab, void* dec_state,
                        const uint8_t* codes, uint16_t* sym_out, int64_t sym_stride, int64_t pos,
                        const uint32_t* win_len, uint32_t* err, cudaStream_t s) {
  if (n <= 0) return;
  note_launch();
  k_dec_search<<<(unsigned)n, kCdfThreads, 0, s>>>(logits, n, V, P, tab, (DecState*)dec_state, codes, sym_out,
                                                   sym_stride, pos, win_len, err);
}

}  // namespace lmgc

// ------------------------------------------------------------------------------------------
// Restricted alphabet (a variant the paper does not describe): the integer CDF of a position is
// taken over the logits of the na ids the serialisation can emit (ascending), and the coded
// symbol is the token's index among them. One warp per row: lane j holds id alpha.id[j].
// ------------------------------------------------------------------------------------------
namespace lmgc {

constexpr int kAlphaWarps = 8;

// this lane's (start, freq) of the row's restricted CDF (lanes >= na: freq 0)
__device__ __forceinline__ void alpha_cdf_lane(const float* __restrict__ z, const AlphaIds& alpha, int P,
                                               const uint32_t* H, const uint32_t* L, uint32_t& start,
                                               uint32_t& freq) {
  const int lane = threadIdx.x & 31, na = alpha.n;
  const bool in = lane < na;
  const float zj = in ? __ldg(z + alpha.id[lane]) : -INFINITY;
  float m = zj;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  const int a = in ? exp2_code(zj, m) : kAMax;
  const uint32_t e = in ? exp2_from_code(a, H, L) : 0u;
  RowStats st;
  st.m = m;
  st.S = warp_sum((uint64_t)e);
  st.Mq = (1ull << P) - (uint64_t)na;
  st.F = (uint32_t)((st.Mq << 32) / st.S);
  const uint64_t g = in ? gfloor(e, st) : 0ull;
  const uint64_t gall = warp_sum(g);
  // the remainder goes to the lowest index whose exponent code is 0 (the largest e, 2^31)
  const uint32_t top = __ballot_sync(0xffffffffu, in && a == 0);
  const int amax = top ? __ffs(top) - 1 : -1;
  uint32_t f = in ? (uint32_t)(1ull + g + (lane == amax ? st.Mq - gall : 0ull)) : 0u;
  uint32_t inc = f;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  start = inc - f;
  freq = f;
}

// the lane holding token t, or -1 (warp-uniform)
__device__ __forceinline__ int alpha_index(const AlphaIds& alpha, int t) {
  const int lane = threadIdx.x & 31;
  const uint32_t hit = __ballot_sync(0xffffffffu, lane < alpha.n && alpha.id[lane] == t);
  return hit ? __ffs(hit) - 1 : -1;
}

// The pairs of k_cdf_pairs (same modes and output indexing) over the restricted alphabet.
__global__ void __launch_bounds__(32 * kAlphaWarps) k_cdf_pairs_alpha(
    const float* __restrict__ logits, int64_t rows, int V, int P, const uint32_t* __restrict__ tab,
    const uint16_t* __restrict__ tok, int64_t n_tok, int W, int64_t first_win,
    uint32_t* __restrict__ start, uint32_t* __restrict__ freq, int mode, int64_t pair_win0, AlphaIds alpha,
    uint32_t* err) {
  __shared__ uint32_t H[256], L[256];
  for (int i = threadIdx.x; i < 256; i += 32 * kAlphaWarps) {
    H[i] = tab[i];
    L[i] = tab[256 + i];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  for (int64_t r = (int64_t)blockIdx.x * kAlphaWarps + (threadIdx.x >> 5); r < rows;
       r += (int64_t)gridDim.x * kAlphaWarps) {
    int sym;
    int64_t out_idx;
    if (mode == 0) {
      sym = tok[r];
      out_idx = r;
    } else {
      const int64_t wl = r / W;
      const int i = (int)(r - wl * W);
      const int64_t gi = (first_win + wl) * W + i;
      if (gi >= n_tok) continue;  // warp-uniform
      sym = tok[gi];
      out_idx = pair_tile_index(first_win + wl - pair_win0, i, pair_tile_groups(W));
    }
    uint32_t st, fr;
    alpha_cdf_lane(logits + r * (int64_t)V, alpha, P, H, L, st, fr);
    const int s = alpha_index(alpha, sym);
    if (s < 0) {
      if (lane == 0) {
        atomicOr(err, kErrCorrupt);  // a token outside the alphabet cannot be coded
        start[out_idx] = 0;
        freq[out_idx] = 1;
      }
    } else if (lane == s) {
      start[out_idx] = st;
      freq[out_idx] = fr;
    }
  }
}

void launch_cdf_pairs_alpha(const float* logits, int64_t rows, int V, int P, const uint32_t* tab,
                            const uint16_t* tok, int64_t n_tok, int W, int64_t first_win,
                            uint32_t* start, uint32_t* freq, int mode, cudaStream_t s, int64_t pair_win0,
                            const AlphaIds& alpha, uint32_t* err) {
  if (rows <= 0) return;
  const int64_t blocks = std::min<int64_t>((rows + kAlphaWarps - 1) / kAlphaWarps, 152 * 16);
  note_launch();
  k_cdf_pairs_alpha<<<(unsigned)blocks, 32 * kAlphaWarps, 0, s>>>(logits, rows, V, P, tab, tok, n_tok, W, first_win,
                                                                 start, freq, mode, pair_win0, alpha,
                                                                 err);
}

// k_dec_search over the restricted alphabet: one warp per decoding window.
__global__ void __launch_bounds__(32 * kAlphaWarps) k_dec_search_alpha(
    const float* __restrict__ logits, int64_t n, int V, int P, const uint32_t* __restrict__ tab,
    DecState* __restrict__ states, const uint8_t* __restrict__ codes, uint16_t* __restrict__ sym_out,
    int64_t sym_stride, int64_t pos, const uint32_t* __restrict__ win_len, AlphaIds alpha, uint32_t* err) {
  __shared__ uint32_t H[256], L[256];
  for (int i = threadIdx.x; i < 256; i += 32 * kAlphaWarps) {
    H[i] = tab[i];
    L[i] = tab[256 + i];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t w = (int64_t)blockIdx.x * kAlphaWarps + (threadIdx.x >> 5);
  if (w >= n || (int64_t)win_len[w] <= pos) return;  // warp-uniform
  DecState s = states[w];
  const uint64_t r = s.R >> P;
  const uint64_t t = s.D / r;
  uint32_t st, fr;
  alpha_cdf_lane(logits + w * (int64_t)V, alpha, P, H, L, st, fr);
  const uint32_t hit = __ballot_sync(0xffffffffu, fr > 0 && (uint64_t)st <= t && t < (uint64_t)st + fr);
  int j = hit ? __ffs(hit) - 1 : -1;
  uint64_t lo = __shfl_sync(0xffffffffu, (uint64_t)st, j < 0 ? 0 : j);
  uint64_t f = __shfl_sync(0xffffffffu, (uint64_t)fr, j < 0 ? 0 : j);
  if (lane != 0) return;
  if (t >= (1ull << P) || j < 0) {
    atomicOr(err, kErrCorrupt);
    j = 0;
    lo = 0;
    f = 1;
  }
  s.D -= r * lo;
  s.R = r * f;
  int k = __clzll((long long)s.R) - 2;
  if (k < 0) k = 0;
  const uint8_t* code = codes + s.code_off;
  for (int i = 0; i < k; i++) s.D = (s.D << 1) | code_bit(code, s.nbits, s.bitpos + i);
  s.bitpos += k;
  s.R <<= k;
  states[w] = s;
  sym_out[w * sym_stride + pos] = alpha.id[j];
}

void launch_dec_search_alpha(const float* logits, int64_t n, int V, int P, const uint32_t* tab, void* dec_state,
                             const uint8_t* codes, uint16_t* sym_out, int64_t sym_stride, int64_t pos,
                             const uint32_t* win_len, const AlphaIds& alpha, uint32_t* err, cudaStream_t s) {
  if (n <= 0) return;
  note_launch();
  k_dec_search_alpha<<<(unsigned)((n + kAlphaWarps - 1) / kAlphaWarps), 32 * kAlphaWarps, 0, s>>>(
      logits, n, V, P, tab, (DecState*)dec_state, codes, sym_out, sym_stride, pos, win_len, alpha, err);
}

}  // namespace lmgc
