// attn_tc.cu -- causal softmax attention of the LM prior (Eq. 2's Llama decoder) on the
// 5th-generation tensor cores, fp16 inputs and probabilities, fp32 softmax and accumulation.
//
// One CTA per (128 query rows, query head, window); 256 threads:
//   warp 0      TMA: the Q tile once, then 64-key K blocks into a 3-stage ring (a stage is reused
//               once the S that read it is done)
//   warp 6      TMA: 64-key V blocks into a 2-stage ring (reused once its P V is done)
//   warp 1      TMEM allocation; one lane issues S = Q K^T (M 128, N 64) two blocks ahead into a
//               3-deep ring in TMEM and commits to the S-done barriers
//   warp 7      one lane issues O += P V (M 128, N hd, V as an MN-major operand; O stays in TMEM
//               for the whole key loop) and commits to the P V-done barriers
// Issuing an MMA, committing and waiting on a barrier each cost tens to a hundred cycles in the
// issuing thread; with small N (64) the two MMA streams are split over two warps so that neither
// chain, rather than the tensor core or the softmax, sets the pace.
//   warps 2-5   softmax: thread i owns query row i (TMEM lane i), so row max and row sum are
//               per-thread loops; P is written as fp16 pairs back into the first 32 columns of
//               the block's own S buffer in TMEM, and the P V MMA reads its A operand from there.
// S(kb+2) reuses the S buffer of block kb-1, so the issuer first waits for P V(kb-1), which read
// P(kb-1) from it.
// Online softmax with a lazily moved reference: P = 2^((s - m) log2(e)/sqrt(hd)) uses the row's
// reference m, which is set to the block maximum on the row's first block and moves again only
// when a block's P sum against the current reference would exceed 2^12 (so P <= 2^12 in fp16);
// the block is then recomputed, and the row of O in TMEM (and the row sum l) is scaled by
// 2^((m_old - m_new) log2(e)/sqrt(hd)) after the previous block's P V has completed. O / l is the
// same softmax whatever the reference, and most blocks need neither a maximum nor a correction.
// Key blocks are 64-aligned and visited in order 0, 1, ...; a block whose keys all lie past a
// row's position leaves that row's state exactly unchanged (no move, P = 0). A decode step
// (one query row per window, keys from the cache) therefore reproduces the prefill row bit for
// bit: the tensor cores' row results do not depend on the other rows of the tile.
// Every mbarrier wait is bounded (~2 s), after which kErrLimit is recorded and the loops end.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "lmgc_internal.cuh"

namespace lmgc {
namespace attn {

constexpr int BQ = 128;
constexpr int kThreads = 256;  // K TMA warp, S-MMA warp, 4 softmax warps, V TMA warp, PV-MMA warp
constexpr float kMaxBlockSum = 4096.f;  // the reference moves when a block's P sum would exceed 2^12

template <int HD>
struct Shape {
  // keys per block: 64 at hd 64 (two CTAs per SM fit in tensor memory), 128 at hd 128, where
  // S = Q K^T then runs as MMAs of N = 128 (half as many MMA issues per key) and the softmax's
  // per-block costs (barrier waits, tensor-memory round trips, the arrive) cover twice the keys
  static constexpr int BKV = 64;
  static constexpr int NS = HD == 128 ? 2 : 3;          // S buffers: S(kb) is issued NS - 1 blocks ahead
  static constexpr int KCH = HD / 64;                   // 64-column (128-byte) chunks of a row
  static constexpr uint32_t Q_BYTES = BQ * HD * 2;
  static constexpr uint32_t KV_CHUNK = BKV * 128;       // one BKV x 64 fp16 chunk
  static constexpr uint32_t K_BYTES = BKV * HD * 2;
  static constexpr uint32_t V_BYTES = BKV * HD * 2;
  static constexpr int KSK = NS, KSV = 2;               // stages of the K ring (one per S buffer) and of the V ring
  static constexpr uint32_t TMEM_S = 0;                 // S ring: NS x BKV columns (P in the first BKV / 2 of each)
  static constexpr uint32_t TMEM_O = NS * BKV;          // O: HD columns (192 at hd 64, 128 at hd 128)
  static constexpr uint32_t TMEM_COLS = 256;            // two CTAs per SM
  static constexpr size_t SMEM = Q_BYTES + KSK * K_BYTES + KSV * V_BYTES + 1024 + 256 + 3 * 1024;
  // S: M 128, N 64; PV: M 128, N HD, B (V) MN-major (bit 16)
  static constexpr uint32_t IDESC_S = (1u << 4) | ((uint32_t)(BKV >> 3) << 17) |
                                      ((uint32_t)(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_PV = (1u << 4) | (1u << 16) |
                                       ((uint32_t)(HD >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t a) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(a), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, uint32_t* err) {
  if (mbar_try(a, parity)) return true;
  const uint64_t t0 = gtimer();
  for (uint32_t i = 1; i < (1u << 28); ++i) {
    if (mbar_try(a, parity)) return true;
    if ((i & 127) == 0 && gtimer() - t0 > 2000000000ull) break;
  }
  atomicOr(err, kErrLimit);
  return false;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t mbar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          dst),
      "l"((uint64_t)map), "r"(mbar), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint32_t mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar) : "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(
          d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D (+)= A B with A read from tensor memory: row i in lane i, two fp16 per 32-bit column, K step
// k of 16 at column offset 8k
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(
          d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// K-major operand, 128-byte swizzle: 8-row groups 1024 B apart (SBO), LBO unused.
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// MN-major operand, 128-byte swizzle: 64-element MN chunks `lbo` bytes apart (LBO), 8-row K
// groups 1024 B apart (SBO).
__device__ __forceinline__ uint64_t desc_mnmajor(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// packed pairs of fp32 (Blackwell's two-wide FMA / ADD: each lane an IEEE round-to-nearest op)
__device__ __forceinline__ uint64_t f2pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2unpack(uint64_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// max of three (one instruction on sm_100 and later)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
// 2^x on the special-function unit (flushes subnormal results to zero; ex2(-inf) = 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// tcgen05.ld without the wait (several loads may be in flight; then tmem_wait())
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// 32 lanes x 32 columns of 32-bit back to TMEM (thread i writes lane base + i)
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
      "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

struct Params {
  __half* out;
  int64_t out_stride;    // elements per output row
  int64_t q_win_stride;  // query rows per window in the q buffer (W prefill, 1 decode)
  int64_t pos_first;     // position of the first query row of a window
  int n_pos;             // query positions per window
  int W;                 // keys rows per window in the kv buffer
  int nq, nkv;
  int q_col0, k_col0, v_col0;  // column offsets of q head 0, k head 0, v head 0
  float scale_log2;            // log2(e) / sqrt(hd)
  uint32_t* err;
  // decode packing: > 0 when each CTA takes the single query row (position pos_first) of every
  // one of the `packed` query heads of KV head blockIdx.y, one per tile row
  int packed;
};

template <int HD, bool PACKED>
__global__ void __launch_bounds__(kThreads, 2)
    k_attn_tc(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tkv, Params p) {
  using S = Shape<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t sq = smem_u32(smem);
  const uint32_t sk = sq + S::Q_BYTES;                // K ring
  const uint32_t sv = sk + S::KSK * S::K_BYTES;        // V ring
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (sv + S::KSV * S::V_BYTES - sq));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 24);
  // barriers, per S buffer i = kb % NS: 0 Q loaded | 1-3 S(kb) ready | 4-6 P(kb) written (128
  //   arrivals) | 7-9 P V(kb) done | 10-12 K stage loaded | 15-16 V stage (kb % 2) loaded.
  // Waits go by the parity of a block's phase, (kb / NS) & 1 (V: (kb / 2) & 1). Such a wait is
  // sound when the previous phase of the barrier has completed and the next cannot complete
  // before the waiter moves on; the comments at each wait say why both hold.
  const uint32_t b_q = smem_u32(bars + 0);
  auto b_s = [&](int i) { return smem_u32(bars + 1 + i); };
  auto b_p = [&](int i) { return smem_u32(bars + 4 + i); };
  auto b_pv = [&](int i) { return smem_u32(bars + 7 + i); };
  auto b_kfull = [&](int i) { return smem_u32(bars + 10 + i); };
  auto b_vfull = [&](int i) { return smem_u32(bars + 15 + i); };
  constexpr int BKV = S::BKV, NS = S::NS;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y;  // query head; with packing, the KV head
  const int64_t w = blockIdx.z;
  const int kvh = PACKED ? h : h / (p.nq / p.nkv);
  // heavy (late) query tiles first
  const int qb = (int)gridDim.x - 1 - (int)blockIdx.x;
  const int64_t pos0 = p.pos_first + (int64_t)qb * BQ;  // position of tile row 0
  const int64_t rem = p.pos_first + p.n_pos - pos0;
  const int nrows = PACKED ? p.packed : (rem < BQ ? (int)rem : BQ);  // valid rows
  const int64_t last_pos = PACKED ? pos0 : pos0 + nrows - 1;
  const int nkb = (int)(last_pos / S::BKV) + 1;
  const int q_row0 = (int)(w * p.q_win_stride + (pos0 - p.pos_first));
  const int kv_row0 = (int)(w * p.W);

  if (PACKED) {
    // rows past the packed ones read zeros (their scores are then finite and need no moves)
    uint4* q4 = reinterpret_cast<uint4*>(smem);
    for (int i = threadIdx.x; i < S::KCH * BQ * 8; i += kThreads)
      if ((i / 8) % BQ >= nrows) q4[i] = make_uint4(0u, 0u, 0u, 0u);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < 19; i++) mbar_init(smem_u32(bars + i), (i >= 4 && i <= 6) ? 128 : 1);  // 13-14, 17-18 unused
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(S::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer: Q, then K blocks ----------------
    if (lane == 0) {
      if (PACKED) {
        // one 128-byte row per head and chunk (the tensor map's box is one row high)
        mbar_expect_tx(b_q, (uint32_t)nrows * S::KCH * 128);
        for (int j = 0; j < nrows; j++)
#pragma unroll
          for (int c = 0; c < S::KCH; c++)
            tma_load_2d(sq + c * (BQ * 128) + j * 128, &tq, b_q, p.q_col0 + (kvh * nrows + j) * HD + 64 * c, q_row0);
      } else {
        mbar_expect_tx(b_q, S::Q_BYTES);
#pragma unroll
        for (int c = 0; c < S::KCH; c++) tma_load_2d(sq + c * (BQ * 128), &tq, b_q, p.q_col0 + h * HD + 64 * c, q_row0);
      }
    }
    __syncwarp();
    for (int kb = 0; kb < nkb; kb++) {
      const int ks = kb % S::KSK;  // == kb % NS, the S buffer index of block kb
      // stage free once S(kb - NS), which read it, is done (this warp saw S(kb - 2 NS) done, and
      // S(kb) needs the stage it is about to load)
      if (kb >= S::KSK &&
          !__all_sync(0xffffffffu, mbar_wait(b_s(ks), (uint32_t)((kb - S::KSK) / NS) & 1u, p.err)))
        break;
      if (lane == 0) {
        mbar_expect_tx(b_kfull(ks), S::K_BYTES);
#pragma unroll
        for (int c = 0; c < S::KCH; c++)
          tma_load_2d(sk + ks * S::K_BYTES + c * S::KV_CHUNK, &tkv, b_kfull(ks), p.k_col0 + kvh * HD + 64 * c,
                      kv_row0 + kb * BKV);
      }
      __syncwarp();
    }
  } else if (warp == 6) {
    // ---------------- TMA producer: V blocks ----------------
    for (int kb = 0; kb < nkb; kb++) {
      const int vs = kb % S::KSV;
      // stage free once P V(kb - 2), which read it, is done (P V completes in order and this warp
      // saw P V(kb - 3) done; the next phase of that barrier, P V(kb - 2 + NS), needs V stages
      // this warp has not loaded yet)
      if (kb >= S::KSV && !__all_sync(0xffffffffu, mbar_wait(b_pv((kb - S::KSV) % NS),
                                                             (uint32_t)((kb - S::KSV) / NS) & 1u, p.err)))
        break;
      if (lane == 0) {
        mbar_expect_tx(b_vfull(vs), S::V_BYTES);
#pragma unroll
        for (int c = 0; c < S::KCH; c++)
          tma_load_2d(sv + vs * S::V_BYTES + c * S::KV_CHUNK, &tkv, b_vfull(vs), p.v_col0 + kvh * HD + 64 * c,
                      kv_row0 + kb * BKV);
      }
      __syncwarp();
    }
  } else if (warp == 1) {
    // ---------------- S issuer: S(kb) = Q K(kb)^T two blocks ahead of the softmax ----------------
    bool ok = __all_sync(0xffffffffu, mbar_wait(b_q, 0, p.err));
    for (int kb = 0; kb < nkb && ok; kb++) {
      const int ks = kb % S::KSK, sb = kb % NS;
      // S(kb) overwrites the buffer from which P V(kb - NS) read P(kb - NS) (this warp saw
      // P V(kb - 2 NS) done; the barrier's next phase, P V(kb), needs S(kb))
      if (kb >= NS && !(ok = __all_sync(0xffffffffu, mbar_wait(b_pv(sb), (uint32_t)((kb - NS) / NS) & 1u, p.err))))
        break;
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(b_kfull(ks), (uint32_t)(kb / S::KSK) & 1u, p.err)))) break;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t kbase = sk + ks * S::K_BYTES;
        // S = Q K^T over hd in steps of 16 (32 bytes inside a 128-byte chunk)
#pragma unroll
        for (int k = 0; k < HD / 16; k++) {
          const int c = k >> 2, o = (k & 3) * 32;
          tc_mma(tmem + S::TMEM_S + sb * BKV, desc_kmajor(sq + c * (BQ * 128) + o),
                 desc_kmajor(kbase + c * S::KV_CHUNK + o), S::IDESC_S, k > 0 ? 1u : 0u);
        }
        tc_commit(b_s(sb));
      }
      __syncwarp();
    }
  } else if (warp == 7) {
    // ---------------- P V issuer ----------------
    bool ok = true;
    for (int kb = 0; kb < nkb && ok; kb++) {
      const int sb = kb % NS, vs = kb % S::KSV;
      ok = __all_sync(0xffffffffu, mbar_wait(b_vfull(vs), (uint32_t)(kb / S::KSV) & 1u, p.err));
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(b_p(sb), (uint32_t)(kb / NS) & 1u, p.err));
      if (!ok) break;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t vbase = sv + vs * S::V_BYTES;
        // O += P V over the block's keys in steps of 16: P (in TMEM) advances 8 columns, V
        // advances 16 rows (2 KiB)
#pragma unroll
        for (int k = 0; k < BKV / 16; k++)
          tc_mma_ts(tmem + S::TMEM_O, tmem + S::TMEM_S + sb * BKV + 8 * k, desc_mnmajor(vbase + k * 2048, S::KV_CHUNK),
                    S::IDESC_PV, (kb > 0 || k > 0) ? 1u : 0u);
        tc_commit(b_pv(sb));
      }
      __syncwarp();
    }
  } else {
    // ---------------- softmax (warps 2..5): thread r owns query row r = TMEM lane r ----------------
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const int pos0_i = (int)pos0, qpos_i = PACKED ? (int)pos0 : (int)pos0 + r;
    // with packing, a warp whose rows are all past the packed ones only keeps the barrier
    // protocol: it waits for each block's S (so its P arrivals stay in phase) and arrives without
    // computing P
    const bool live = !PACKED || q4 * 32 < nrows;
    const uint32_t tl = (uint32_t)(q4 * 32) << 16;
    const float c = p.scale_log2;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int kb = 0; kb < nkb; kb++) {
      const int sb = kb % NS;
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(b_s(sb), (uint32_t)(kb / NS) & 1u, p.err)))) break;
      if (!live) {
        mbar_arrive(b_p(sb));
        continue;
      }
      tc_fence_after();
      float s[BKV];
      // S row of this block into s[], causally masked (only on blocks that reach past the tile's
      // first position)
      auto load_s = [&]() {
        // every 32-column load of the row in flight, then one wait
        uint32_t a[BKV / 32][32];
#pragma unroll
        for (int q = 0; q < BKV / 32; q++) tmem_ld32_nowait(tmem + tl + S::TMEM_S + sb * BKV + 32 * q, a[q]);
        tmem_wait();
#pragma unroll
        for (int q = 0; q < BKV / 32; q++)
#pragma unroll
          for (int j = 0; j < 32; j++) s[32 * q + j] = __uint_as_float(a[q][j]);
        if ((int)(kb * BKV + BKV - 1) > pos0_i) {
#pragma unroll
          for (int j = 0; j < BKV; j++)
            if (kb * BKV + j > qpos_i) s[j] = -INFINITY;
        }
      };
      // s[j] <- 2^((s[j] - m) c) in place; returns the block's sum (fixed order)
      auto exp_block = [&]() -> float {
        const float nb = -m * c;
        const uint64_t c2 = f2pack(c, c), nb2 = f2pack(nb, nb);
        uint64_t acc0 = 0ull, acc1 = 0ull;  // (+0, +0) packed
#pragma unroll
        for (int j = 0; j < BKV; j += 2) {
          float t0, t1;
          f2unpack(ffma2(f2pack(s[j], s[j + 1]), c2, nb2), t0, t1);
          s[j] = ex2_approx(t0);
          s[j + 1] = ex2_approx(t1);
          if ((j >> 1) & 1) acc1 = fadd2(acc1, f2pack(s[j], s[j + 1]));
          else acc0 = fadd2(acc0, f2pack(s[j], s[j + 1]));
        }
        float a0, a1, a2, a3;
        f2unpack(acc0, a0, a1);
        f2unpack(acc1, a2, a3);
        return (a0 + a1) + (a2 + a3);
      };
      load_s();
      // Common case: P against the current reference. The reference moves (to the block
      // maximum) on a row's first block and whenever the block's P sum would exceed 2^12 (or is
      // not finite); the block is then recomputed. A warp takes that path if any of its rows
      // needs it, and its other rows recompute the same values.
      float bsum = 0.f;
      if (kb > 0) bsum = exp_block();
      const bool move = kb == 0 || !(bsum <= kMaxBlockSum);
      if (__any_sync(0xffffffffu, move)) {
        if (kb > 0) load_s();
        float corr = 1.f;
        if (move) {
          float mx4[4];
#pragma unroll
          for (int i = 0; i < 4; i++) mx4[i] = s[i];
#pragma unroll
          for (int j = 4; j < BKV; j += 2) mx4[(j >> 1) & 3] = fmax3(mx4[(j >> 1) & 3], s[j], s[j + 1]);
          const float mx = fmaxf(fmax3(mx4[0], mx4[1], mx4[2]), mx4[3]);  // finite: key 0 is unmasked
          corr = kb == 0 ? 0.f : ex2_approx((m - mx) * c);
          l *= corr;
          m = mx;
        }
        if (kb > 0) {
          // scale this warp's rows of O (factor 1 for rows that did not move) once the previous
          // block's P V has landed in TMEM (P V(kb - 1 - NS) has completed, as S(kb) has; the
          // barrier's next phase, P V(kb - 1 + NS), needs P from these warps)
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(b_pv((kb - 1) % NS), (uint32_t)((kb - 1) / NS) & 1u, p.err))))
            break;
          tc_fence_after();
#pragma unroll 1
          for (int cc = 0; cc < HD / 32; cc++) {
            uint32_t o[32];
            tmem_ld32_nowait(tmem + tl + S::TMEM_O + cc * 32, o);
            tmem_wait();
#pragma unroll
            for (int j = 0; j < 32; j++) o[j] = __float_as_uint(__uint_as_float(o[j]) * corr);
            tmem_st32(tmem + tl + S::TMEM_O + cc * 32, o);
          }
          tmem_st_wait();
        }
        bsum = exp_block();
      }
      l += bsum;
      // P as fp16 pairs over the first BKV / 2 columns of this block's S buffer (already read)
#pragma unroll
      for (int h2 = 0; h2 < BKV / 2; h2 += 32) {
        uint32_t pw[32];
#pragma unroll
        for (int j = 0; j < 32; j++) {
          __half2 hb = __floats2half2_rn(s[2 * (h2 + j)], s[2 * (h2 + j) + 1]);
          pw[j] = *reinterpret_cast<uint32_t*>(&hb);
        }
        tmem_st32(tmem + tl + S::TMEM_S + sb * BKV + h2, pw);
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(b_p(sb));
    }
    // O / l once the last P V has completed (S(last) implies P V(last - NS), the previous phase of
    // P V(last)'s barrier and, as P V completes in order, of P V(last - 1)'s)
    for (int j = nkb >= 2 ? nkb - 2 : 0; j < nkb && ok; j++)
      ok = __all_sync(0xffffffffu, mbar_wait(b_pv(j % NS), (uint32_t)(j / NS) & 1u, p.err));
    if (ok && live) {
      tc_fence_after();
      const float inv = 1.f / l;
      __half* dst = PACKED ? p.out + (int64_t)q_row0 * p.out_stride + (int64_t)(kvh * nrows + r) * HD
                             : p.out + ((int64_t)q_row0 + r) * p.out_stride + (int64_t)h * HD;
#pragma unroll 1
      for (int cc = 0; cc < HD / 32; cc++) {
        uint32_t o[32];
        tmem_ld32_nowait(tmem + tl + S::TMEM_O + cc * 32, o);
        tmem_wait();
        if (r < nrows) {
#pragma unroll
          for (int q = 0; q < 4; q++) {
            uint32_t wv[4];
#pragma unroll
            for (int t = 0; t < 4; t++) {
              __half2 hb = __floats2half2_rn(__uint_as_float(o[8 * q + 2 * t]) * inv,
                                             __uint_as_float(o[8 * q + 2 * t + 1]) * inv);
              wv[t] = *reinterpret_cast<uint32_t*>(&hb);
            }
            reinterpret_cast<uint4*>(dst + cc * 32)[q] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(S::TMEM_COLS) : "memory");
  }
}

static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static std::once_flag g_once;

static void init_once() {
  cudaDriverEntryPointQueryResult q;
  void* fn = nullptr;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  int dev = 0, major = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (major != 10) g_encode = nullptr;
  cudaFuncSetAttribute(k_attn_tc<64, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<64>::SMEM);
  cudaFuncSetAttribute(k_attn_tc<128, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<128>::SMEM);
  cudaFuncSetAttribute(k_attn_tc<64, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<64>::SMEM);
  cudaFuncSetAttribute(k_attn_tc<128, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Shape<128>::SMEM);
}

static bool make_map(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace attn

bool tc_attention_supported(int hd, int64_t qkv_dim) {
  std::call_once(attn::g_once, attn::init_once);
  return attn::g_encode != nullptr && (hd == 64 || hd == 128) && qkv_dim % 64 == 0;
}

void launch_attention_tc(const void* q, int64_t q_rows, int64_t q_dim, const void* kv, int64_t kv_rows,
                         int64_t kv_dim, int k_off, int v_off, void* out, int64_t out_stride, int nq, int nkv, int hd,
                         int W, int64_t n_win, int64_t pos_first, int n_pos, int64_t q_win_stride, uint32_t* err,
                         cudaStream_t s) {
  using namespace attn;
  std::call_once(g_once, init_once);
  CUtensorMap tq, tkv;
  if (!make_map(&tq, q, (uint64_t)q_dim, (uint64_t)q_rows, BQ) ||
      !make_map(&tkv, kv, (uint64_t)kv_dim, (uint64_t)kv_rows, hd == 128 ? Shape<128>::BKV : Shape<64>::BKV)) {
    set_thread_error("cuTensorMapEncodeTiled failed (attention)");
    return;
  }
  Params p;
  p.out = (__half*)out;
  p.out_stride = out_stride;
  p.q_win_stride = q_win_stride;
  p.pos_first = pos_first;
  p.n_pos = n_pos;
  p.W = W;
  p.nq = nq;
  p.nkv = nkv;
  p.q_col0 = 0;
  p.k_col0 = k_off;
  p.v_col0 = v_off;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)hd));
  p.err = err;
  // a decode step (one query row per window) packs the query heads of each KV head into one tile
  const int group = nq / nkv;
  p.packed = (n_pos == 1 && q_win_stride == 1 && group > 1 && group <= 32) ? group : 0;
  if (p.packed && !make_map(&tq, q, (uint64_t)q_dim, (uint64_t)q_rows, 1)) {
    set_thread_error("cuTensorMapEncodeTiled failed (attention)");
    return;
  }
  dim3 grid((unsigned)((n_pos + BQ - 1) / BQ), (unsigned)(p.packed ? nkv : nq), (unsigned)n_win);
  note_launch();
  if (p.packed) {
    if (hd == 64) k_attn_tc<64, true><<<grid, kThreads, Shape<64>::SMEM, s>>>(tq, tkv, p);
    else k_attn_tc<128, true><<<grid, kThreads, Shape<128>::SMEM, s>>>(tq, tkv, p);
  } else {
    if (hd == 64) k_attn_tc<64, false><<<grid, kThreads, Shape<64>::SMEM, s>>>(tq, tkv, p);
    else k_attn_tc<128, false><<<grid, kThreads, Shape<128>::SMEM, s>>>(tq, tkv, p);
  }
}

}  // namespace lmgc
