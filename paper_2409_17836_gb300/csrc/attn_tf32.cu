// attn_tf32.cu -- causal softmax attention of an fp32 model (Eq. 2's Llama decoder, head dim
// 32 or 64) on the 5th-generation tensor cores in three-pass TF32 form, fp32 softmax.
//
// S = Q K^T and O += P V are tcgen05 MMAs of kind::tf32 with every operand split as x = hi + lo
// (hi: x with its low 13 bits cleared) and lo_A hi_B + hi_A lo_B + hi_A hi_B accumulated in fp32
// in tensor memory (see gemm_tf32.cu for the error terms). All operands are K-major in shared
// memory with the 128-byte swizzle: Q and K as TMA lands them (split in place); V transposed to
// [hd][keys] while it is split; P written by the softmax threads.
//
// One CTA per (128 query rows, query head, window), 128 threads, thread r owning query row r
// (TMEM lane r). Per 64-key block, in order: TMA of K and V, split, S MMAs, the row's online
// softmax (running maximum m and sum l; O in TMEM rescaled by 2^((m_old - m_new) log2(e)/sqrt(hd))
// when m moves), P split into shared memory, P V MMAs. The steps run one after another (no
// warp specialisation): fp32 models are the small configuration, where this kernel takes
// microseconds. A block whose keys all lie past a row's position leaves that row's m, l and O
// exactly unchanged (P = 0, scale 1), so a decode step (one query row per window, keys from the
// cache) reproduces the prefill row bit for bit. Every mbarrier wait is bounded (~2 s).
#include "tf32_common.cuh"

namespace lmgc {
namespace tf32 {
namespace attn {

constexpr int BQ = 128, BKV = 64, kThreads = 128;

template <int HD>
struct Shape {
  static constexpr int KCH = HD / 32;                 // 128-byte chunks of a Q or K row
  static constexpr uint32_t Q_BYTES = BQ * HD * 4;
  static constexpr uint32_t KV_BYTES = BKV * HD * 4;
  static constexpr uint32_t P_BYTES = BQ * BKV * 4;
  // shared memory: Q | Q lo | K | K lo | V as landed | V^T | V^T lo | P | P lo
  static constexpr uint32_t OFF_QLO = Q_BYTES, OFF_K = 2 * Q_BYTES, OFF_KLO = OFF_K + KV_BYTES,
                            OFF_V = OFF_KLO + KV_BYTES, OFF_VT = OFF_V + KV_BYTES, OFF_VTLO = OFF_VT + KV_BYTES,
                            OFF_P = OFF_VTLO + KV_BYTES, OFF_PLO = OFF_P + P_BYTES, OFF_BAR = OFF_PLO + P_BYTES;
  static constexpr size_t SMEM = OFF_BAR + 64 + 1024;
  static constexpr uint32_t TMEM_S = 0, TMEM_O = BKV, TMEM_COLS = 128;
  // kind::tf32, D fp32, A and B TF32, both K-major: S is M 128 x N 64, P V is M 128 x N hd
  static constexpr uint32_t IDESC_S =
      (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(BKV >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_PV =
      (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(HD >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
};

struct Params {
  float* out;
  int64_t out_stride;    // elements per output row
  int64_t q_win_stride;  // query rows per window in the q buffer (W prefill, 1 decode)
  int64_t pos_first;     // position of the first query row of a window
  int n_pos;             // query positions per window
  int W;                 // key rows per window in the kv buffer
  int nq, nkv;
  int k_col0, v_col0;    // column offsets of k head 0 and v head 0 in the kv buffer
  float scale_log2;      // log2(e) / sqrt(hd)
  uint32_t* err;
};

// the three MMA streams of one product over k_steps 8-wide K slices of K-major operands whose
// 32-float chunks are chunk_a / chunk_b bytes apart
__device__ __forceinline__ void mma3(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint32_t chunk_a, uint32_t b_hi,
                                     uint32_t b_lo, uint32_t chunk_b, int k_steps, uint32_t idesc, bool acc0) {
  for (int k = 0; k < k_steps; k++) {
    const uint32_t oa = (uint32_t)(k >> 2) * chunk_a + 32u * (uint32_t)(k & 3);
    const uint32_t ob = (uint32_t)(k >> 2) * chunk_b + 32u * (uint32_t)(k & 3);
    tc_mma(d, desc_kmajor(a_lo + oa), desc_kmajor(b_hi + ob), idesc, (acc0 || k > 0) ? 1u : 0u);
    tc_mma(d, desc_kmajor(a_hi + oa), desc_kmajor(b_lo + ob), idesc, 1u);
    tc_mma(d, desc_kmajor(a_hi + oa), desc_kmajor(b_hi + ob), idesc, 1u);
  }
}

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
    k_attn_tf32(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tkv, Params p) {
  using S = Shape<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);  // 0 TMA landed | 1 MMAs done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 4);
  const uint32_t b_tma = smem_u32(bars + 0), b_mma = smem_u32(bars + 1);
  const uint32_t s0 = smem_u32(smem);

  const int t = threadIdx.x, warp = t >> 5;
  const int h = blockIdx.y;
  const int64_t w = blockIdx.z;
  const int kvh = h / (p.nq / p.nkv);
  const int qb = (int)gridDim.x - 1 - (int)blockIdx.x;  // heavy (late) query tiles first
  const int64_t pos0 = p.pos_first + (int64_t)qb * BQ;
  const int64_t rem = p.pos_first + p.n_pos - pos0;
  const int nrows = rem < BQ ? (int)rem : BQ;
  const int64_t last_pos = pos0 + nrows - 1;
  const int nkb = (int)(last_pos / BKV) + 1;
  const int q_row0 = (int)(w * p.q_win_stride + (pos0 - p.pos_first));
  const int kv_row0 = (int)(w * p.W);
  const int64_t qpos = pos0 + t;

  if (t == 0) {
    mbar_init(b_tma, 1);
    mbar_init(b_mma, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(S::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tl = (uint32_t)(warp * 32) << 16;  // this warp's TMEM lanes
  uint32_t ph_tma = 0, ph_mma = 0;
  bool ok = true;

  // Q (rows past the window's last position are read as whatever follows; their results are
  // discarded), split in place
  if (t == 0) {
    mbar_expect_tx(b_tma, S::Q_BYTES);
#pragma unroll
    for (int c = 0; c < S::KCH; c++) tma_load_2d(s0 + c * (BQ * 128), &tq, b_tma, h * HD + 32 * c, q_row0);
  }
  ok = __syncthreads_and(mbar_wait(b_tma, ph_tma, p.err));
  ph_tma ^= 1u;
  if (ok) split_tile(smem, S::OFF_QLO, (int)(S::Q_BYTES / 16), t);

  const float c = p.scale_log2;
  float m = -INFINITY, l = 0.f;
  for (int kb = 0; kb < nkb && ok; kb++) {
    // K and V of the block
    if (t == 0) {
      mbar_expect_tx(b_tma, 2 * S::KV_BYTES);
#pragma unroll
      for (int cc = 0; cc < S::KCH; cc++) {
        tma_load_2d(s0 + S::OFF_K + cc * (BKV * 128), &tkv, b_tma, p.k_col0 + kvh * HD + 32 * cc, kv_row0 + kb * BKV);
        tma_load_2d(s0 + S::OFF_V + cc * (BKV * 128), &tkv, b_tma, p.v_col0 + kvh * HD + 32 * cc, kv_row0 + kb * BKV);
      }
    }
    if (!(ok = __syncthreads_and(mbar_wait(b_tma, ph_tma, p.err)))) break;
    ph_tma ^= 1u;
    split_tile(smem + S::OFF_K, S::KV_BYTES, (int)(S::KV_BYTES / 16), t);
    // V [key][d] (as landed) -> V^T [d][key] hi and lo, K-major over the keys
    for (int e = t; e < BKV * HD; e += kThreads) {
      const int j = e / HD, d = e - j * HD;
      const float v = *reinterpret_cast<const float*>(smem + S::OFF_V + sw128_offset(j, d, BKV));
      const float hi = tf32_hi(v);
      const uint32_t o = sw128_offset(d, j, HD);
      *reinterpret_cast<float*>(smem + S::OFF_VT + o) = hi;
      *reinterpret_cast<float*>(smem + S::OFF_VTLO + o) = __fsub_rn(v, hi);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    // S = Q K^T
    if (t == 0) {
      tc_fence_after();
      mma3(tmem + S::TMEM_S, s0, s0 + S::OFF_QLO, BQ * 128, s0 + S::OFF_K, s0 + S::OFF_KLO, BKV * 128, HD / 8,
           S::IDESC_S, false);
      tc_commit(b_mma);
    }
    if (!(ok = __syncthreads_and(mbar_wait(b_mma, ph_mma, p.err)))) break;
    ph_mma ^= 1u;
    tc_fence_after();
    float s[BKV];
    {
      uint32_t r0[32], r1[32];
      tmem_ld32(tmem + tl + S::TMEM_S, r0);
      tmem_ld32(tmem + tl + S::TMEM_S + 32, r1);
#pragma unroll
      for (int j = 0; j < 32; j++) {
        s[j] = __uint_as_float(r0[j]);
        s[32 + j] = __uint_as_float(r1[j]);
      }
    }
    // causal mask, block maximum, and the row's online softmax state
    float bm = -INFINITY;
#pragma unroll
    for (int j = 0; j < BKV; j++) {
      if ((int64_t)kb * BKV + j > qpos) s[j] = -INFINITY;
      bm = fmaxf(bm, s[j]);
    }
    float corr = 1.f;
    if (bm > m) {  // the reference moves (always on a row's first block: key 0 is unmasked)
      corr = kb == 0 ? 0.f : exp2f((m - bm) * c);
      m = bm;
    }
    float bsum = 0.f;
#pragma unroll
    for (int j = 0; j < BKV; j++) {
      s[j] = s[j] == -INFINITY ? 0.f : exp2f((s[j] - m) * c);
      bsum += s[j];
    }
    l = l * corr + bsum;
    // O *= corr once the previous P V has completed (it has: its MMAs were waited for); rows
    // whose reference did not move multiply by exactly 1
    if (kb > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
#pragma unroll 1
      for (int cc = 0; cc < HD / 32; cc++) {
        uint32_t o[32];
        tmem_ld32(tmem + tl + S::TMEM_O + 32 * cc, o);
#pragma unroll
        for (int j = 0; j < 32; j++) o[j] = __float_as_uint(__uint_as_float(o[j]) * corr);
        tmem_st32(tmem + tl + S::TMEM_O + 32 * cc, o);
      }
    }
    // P (row t, keys 0..63) split into shared memory, K-major with the 128-byte swizzle
#pragma unroll
    for (int j = 0; j < BKV; j += 4) {
      const uint32_t o = sw128_offset(t, j, BQ);
      float4 hi, lo;
      hi.x = tf32_hi(s[j]);
      hi.y = tf32_hi(s[j + 1]);
      hi.z = tf32_hi(s[j + 2]);
      hi.w = tf32_hi(s[j + 3]);
      lo.x = __fsub_rn(s[j], hi.x);
      lo.y = __fsub_rn(s[j + 1], hi.y);
      lo.z = __fsub_rn(s[j + 2], hi.z);
      lo.w = __fsub_rn(s[j + 3], hi.w);
      *reinterpret_cast<float4*>(smem + S::OFF_P + o) = hi;
      *reinterpret_cast<float4*>(smem + S::OFF_PLO + o) = lo;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    // O += P V
    if (t == 0) {
      tc_fence_after();
      mma3(tmem + S::TMEM_O, s0 + S::OFF_P, s0 + S::OFF_PLO, BQ * 128, s0 + S::OFF_VT, s0 + S::OFF_VTLO, HD * 128,
           BKV / 8, S::IDESC_PV, kb > 0);
      tc_commit(b_mma);
    }
    if (!(ok = __syncthreads_and(mbar_wait(b_mma, ph_mma, p.err)))) break;
    ph_mma ^= 1u;
  }
  if (ok) {
    tc_fence_after();
    const float inv = 1.f / l;
#pragma unroll 1
    for (int cc = 0; cc < HD / 32; cc++) {
      uint32_t o[32];
      tmem_ld32(tmem + tl + S::TMEM_O + 32 * cc, o);
      if (t < nrows) {
        float* dst = p.out + ((int64_t)q_row0 + t) * p.out_stride + (int64_t)h * HD + 32 * cc;
#pragma unroll
        for (int j = 0; j < 32; j += 4)
          *reinterpret_cast<float4*>(dst + j) = make_float4(__uint_as_float(o[j]) * inv, __uint_as_float(o[j + 1]) * inv,
                                                            __uint_as_float(o[j + 2]) * inv, __uint_as_float(o[j + 3]) * inv);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(S::TMEM_COLS) : "memory");
  }
}

static std::once_flag g_once;
static bool g_ready = false;

static void init_once() {
  if (!encoder()) return;
  cudaFuncSetAttribute(k_attn_tf32<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<32>::SMEM);
  cudaFuncSetAttribute(k_attn_tf32<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<64>::SMEM);
  g_ready = true;
}

}  // namespace attn
}  // namespace tf32

bool tf32_attention_supported(int hd, int64_t q_dim, int64_t kv_dim) {
  std::call_once(tf32::attn::g_once, tf32::attn::init_once);
  return tf32::attn::g_ready && (hd == 32 || hd == 64) && q_dim % 32 == 0 && kv_dim % 32 == 0;
}

void launch_attention_tf32(const float* q, int64_t q_rows, int64_t q_dim, const float* kv, int64_t kv_rows,
                           int64_t kv_dim, int k_off, int v_off, float* out, int64_t out_stride, int nq, int nkv,
                           int hd, int W, int64_t n_win, int64_t pos_first, int n_pos, int64_t q_win_stride,
                           uint32_t* err, cudaStream_t s) {
  using namespace tf32;
  using namespace tf32::attn;
  std::call_once(g_once, init_once);
  if (n_win <= 0 || n_pos <= 0) return;
  CUtensorMap tq, tkv;
  if (!g_ready || !make_map_f32(&tq, q, (uint64_t)q_dim, (uint64_t)q_rows, BQ) ||
      !make_map_f32(&tkv, kv, (uint64_t)kv_dim, (uint64_t)kv_rows, BKV)) {
    set_thread_error("cuTensorMapEncodeTiled failed (tf32 attention)");
    return;
  }
  Params p;
  p.out = out;
  p.out_stride = out_stride;
  p.q_win_stride = q_win_stride;
  p.pos_first = pos_first;
  p.n_pos = n_pos;
  p.W = W;
  p.nq = nq;
  p.nkv = nkv;
  p.k_col0 = k_off;
  p.v_col0 = v_off;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)hd));
  p.err = err;
  dim3 grid((unsigned)((n_pos + BQ - 1) / BQ), (unsigned)nq, (unsigned)n_win);
  note_launch();
  if (hd == 32) k_attn_tf32<32><<<grid, kThreads, Shape<32>::SMEM, s>>>(tq, tkv, p);
  else k_attn_tf32<64><<<grid, kThreads, Shape<64>::SMEM, s>>>(tq, tkv, p);
}

}  // namespace lmgc
