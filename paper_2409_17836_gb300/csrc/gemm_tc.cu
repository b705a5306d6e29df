// gemm_tc.cu -- the model's dense contractions (the linear layers and the vocabulary projection of
// the LM prior, Eq. 2) on the 5th-generation tensor cores: C[M][N] (op)= A[M][K] . B[N][K]^T,
// fp16 operands (the model's bf16-valued weights held exactly in fp16, fp16 activations), fp32
// accumulation in tensor memory.
//
// Persistent, warp-specialised kernel on CTA pairs (clusters of 2, one CTA per SM): a pair computes
// 256x256 output tiles with tcgen05.mma.cta_group::2 (M 256, N 256, K 16). CTA r of the pair
// stages rows [128 r, 128 r + 128) of the tile's A block and rows [128 r, 128 r + 128) of its B
// block (the N dimension), so each SM reads 8 KiB of operands per MMA instead of 12, and holds
// its own 128 output rows in its tensor memory.
//   warp 0      TMA producer (both CTAs): 128x64 A and 128x64 B tiles (128-byte swizzle), two
//               per operand and stage in a 3-stage ring (one in 6 stages for the fp32 logits);
//               both CTAs' copies complete on the leader CTA's full barrier
//   warp 1      both CTAs allocate 512 TMEM columns together; in the leader one lane issues the
//               MMAs and multicasts its commits to both CTAs' empty and accumulator-full barriers
//   warps 2..   epilogue (both CTAs): 4 warps (8 for the fp32 logits, whose stores dominate): warp
//               w reads TMEM lanes 32 (w mod 4) .. and, with 8 warps, one column half of the tile;
//               tcgen05.ld 32 lanes x 32 columns, convert / add, store to global (fp32 outputs
//               through a shared-memory transpose); then arrive on the leader's accumulator-empty
//               barrier
// Two 128x256 fp32 accumulators per CTA (2 x 256 TMEM columns) let the epilogue of one tile run
// under the main loop of the next. Tiles are visited in groups of M-blocks so the A and B tiles
// in flight stay in L2.
//
// Row invariance (needed by the KV-cached decoder): every output element is accumulated over k
// in the same order by the same MMA shape whatever M is; rows past M are zero-filled by TMA and
// never stored.
//
// Every mbarrier wait is bounded (about 2 s of %globaltimer); on expiry the kernel records
// kErrLimit, leaves its loops and still frees its tensor memory.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "lmgc_internal.cuh"

namespace lmgc {
namespace tc {

constexpr int BM = 128;  // rows per CTA; a pair covers 2 BM = 256 rows of a tile
constexpr int BN = 256, BK = 64;
constexpr int TM = 2 * BM;  // tile rows
// epilogue warps per epilogue kind, and the CTA size
template <int EPI>
struct EpiShape {
  // k depth of a ring stage in 64-wide (128-byte swizzle) atoms, and stages: two atoms (8 MMAs
  // per barrier wait and commit, which cost the MMA warp about as much as the MMAs themselves)
  // in 3 stages; the fp32 logits keep one atom in 6 stages (their 8 epilogue warps and
  // streamed weights do better with a finer ring)
  static constexpr int kSub = EPI == kStoreF32 ? 1 : 2;
  static constexpr int kStages = EPI == kStoreF32 ? 6 : 3;
  static constexpr int kWarps = (EPI == kStoreF32 || EPI == kAddResidualWide) ? 8 : 4;
  static constexpr int kThreads = 64 + 32 * kWarps;
  static constexpr uint32_t kStgBytes = kWarps == 8 ? 8 * 32 * 32 * 4 : 4 * 32 * 36 * 4;
};
constexpr bool is_resid(int epi) { return epi == kAddResidual || epi == kAddResidualWide; }
constexpr uint32_t A_SUB = BM * BK * 2;        // 16 KiB per k atom
constexpr uint32_t B_SUB = (BN / 2) * BK * 2;  // 16 KiB per k atom: this CTA's half of the B tile
constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
// tile order: groups of group_m M-blocks (256 rows each), N-blocks swept inside a group (M
// fastest). A weight operand that fits in L2 (<= kKeepBBytes) is read with an evict-last policy;
// its groups are 8 M-blocks for narrow GEMMs and 32 (8192 rows) for wide ones. A larger weight
// streams past the group's A rows, which every N-block of the group re-reads: groups of 16
// (4096 rows) keep them in L2 far better than 32 at K = 4096 (measured on a 1-layer Llama-2-7B
// layer: 16.7 -> 10.7 GB of DRAM traffic), and the lower DRAM power lets the power-capped step
// hold a higher clock (1387 -> 1425 MHz, 1234 -> 1185 ms per Llama-2-7B step).
constexpr int64_t kKeepBBytes = 48ll << 20;
// fp32 epilogue staging: per epilogue warp 32 rows x 32 fp32 columns, laid out so that both the
// row-per-thread writes and the row-per-8-lanes reads take 4 wavefronts per 512 B: with 4 warps a
// row pitch of 36 words; with 8 warps (which need the space) a pitch of 32 words with the 16-byte
// slot j of row r stored at slot j ^ (r mod 8)
template <int NH>
__device__ __forceinline__ int stg_off(int r, int j) {
  return NH == 2 ? r * 32 + ((j ^ (r & 7)) << 2) : r * 36 + (j << 2);
}
template <int EPI>
constexpr size_t smem_bytes() {
  return (size_t)EpiShape<EPI>::kStages * EpiShape<EPI>::kSub * (A_SUB + B_SUB) + 256 + EpiShape<EPI>::kStgBytes +
         1024;
}

// instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A and B f16 (bits 7-9, 10-12 = 0),
// both K-major (15, 16 = 0), N >> 3 at bits 17-22, M >> 4 at bits 24-28 (M = 256: the pair)
constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(TM >> 4) << 24);

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  // the suspend-time hint lets a waiting warp sleep until the phase completes instead of spinning
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(a), "r"(parity), "r"(0x989680u)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// non-blocking probe of a phase: cheaper than try_wait when the phase has already completed
__device__ __forceinline__ bool mbar_test(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(a), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity; false (and kErrLimit) after ~2 s.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, uint32_t* err) {
  if (mbar_test(a, parity) || mbar_try(a, parity)) return true;
  const uint64_t t0 = gtimer();
  for (uint32_t i = 1; i < (1u << 28); ++i) {
    if (mbar_try(a, parity)) return true;
    if ((i & 127) == 0 && gtimer() - t0 > 2000000000ull) break;
  }
  atomicOr(err, kErrLimit);
  return false;
}

// tile copy into this CTA's shared memory that completes on a barrier of either CTA of the pair
// (`mbar` is a shared::cluster address)
__device__ __forceinline__ void tma_load_pair(uint32_t dst, const CUtensorMap* map, uint32_t mbar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(dst),
      "l"((uint64_t)map), "r"(mbar), "r"(x), "r"(y)
      : "memory");
}

// the same with an L2 cache policy (createpolicy) attached to the read
__device__ __forceinline__ void tma_load_pair_hint(uint32_t dst, const CUtensorMap* map, uint32_t mbar, int x, int y,
                                                   uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1, {%3, %4}], [%2], %5;" ::"r"(dst),
      "l"((uint64_t)map), "r"(mbar), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// arrive on the barrier at this offset in both CTAs of the pair once the issued MMAs complete
__device__ __forceinline__ void tc_commit_pair(uint32_t mbar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(mbar),
      "h"((uint16_t)3)
      : "memory");
}
// the same shared-memory offset in CTA `rank` of the cluster (a shared::cluster address)
__device__ __forceinline__ uint32_t cluster_addr(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_a) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_a) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(
          d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(IDESC), "r"(accumulate)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile written by TMA with the 128-byte
// swizzle: rows of 64 bf16 (128 B), 8-row groups 1024 B apart (stride byte offset), leading
// byte offset unused for swizzled K-major layouts, version 1, layout SWIZZLE_128B (2).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// 32 TMEM lanes x 32 columns of 32-bit: thread i of the warp gets lane (base + i), 32 columns.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

struct Params {
  void* C;
  int64_t M, N, K;
  int tiles_m, tiles_n, num_kb;
  int group_m, keep_b;
  uint32_t* err;
  // kQKVRope: rotary embedding of columns [0, rope_cols) in heads of rope_hd; row m sits at
  // position rope_pos0 + m % rope_pos_mod; rope_cs[pos * rope_hd/2 + i] = (cos, sin)
  const float2* rope_cs;
  int rope_cols, rope_hd, rope_pos_mod;
  int64_t rope_pos0;
  // fused RMSNorm of the A rows: when row_ss is set, the result of row m is scaled by
  // rsqrt(sum_k row_ss[m * ss_parts + k] * ss_inv_d + ss_eps) before the epilogue's operation
  const float* row_ss;
  int ss_parts;
  float ss_inv_d, ss_eps;
  // kAddResidual(Wide): also write fp16(x) to xh and the row's sum of squares over each epilogue
  // warp's columns to ss_out[m * tiles_n * NH + nb * NH + hw] (NH = 1, or 2 for the wide form)
  __half* xh;
  float* ss_out;
  // kStoreF32: row_max[m] = max over the launch of float_key(C[m][n]) (atomic; zeroed beforehand)
  uint32_t* row_max;
};

__device__ __forceinline__ float row_scale(const Params& p, int64_t m) {
  if (!p.row_ss || m >= p.M) return 1.f;
  const float* s = p.row_ss + m * p.ss_parts;
  float t = 0.f;
  for (int k = 0; k < p.ss_parts; k++) t += s[k];
  return rsqrtf(t * p.ss_inv_d + p.ss_eps);
}

__device__ __forceinline__ void tile_coords(int t, const Params& p, int& mb, int& nb) {
  const int per_group = p.group_m * p.tiles_n;
  const int g = t / per_group;
  const int first_m = g * p.group_m;
  const int gm = min(p.tiles_m - first_m, p.group_m);
  const int r = t - g * per_group;
  mb = first_m + r % gm;
  nb = r / gm;
}

// L2 prefetch of row m's fp32 residual, columns [n0, n0 + cnt) (N % 32 == 0, n0 % 32 == 0)
__device__ __forceinline__ void prefetch_residual(const Params& p, int64_t m, int64_t n0, int cnt) {
  if (m >= p.M || n0 >= p.N) return;
  const char* xr = reinterpret_cast<const char*>(reinterpret_cast<const float*>(p.C) + m * p.N + n0);
  const int lines = (int)(min((int64_t)cnt, p.N - n0) * 4 / 128);
  for (int j = 0; j < lines; j++) asm volatile("prefetch.global.L2 [%0];" ::"l"(xr + j * 128));
}

template <int EPI>
__device__ __forceinline__ void store_chunk(const Params& p, int64_t m, int64_t n0, const uint32_t (&r)[32]) {
  if (EPI == kStore) {
    __half* c = reinterpret_cast<__half*>(p.C) + m * p.N + n0;
    if (n0 + 32 <= p.N && (p.N & 7) == 0) {
      uint32_t w[16];
#pragma unroll
      for (int j = 0; j < 16; j++) {
        __half2 h = __floats2half2_rn(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
        w[j] = *reinterpret_cast<uint32_t*>(&h);
      }
      uint4* d = reinterpret_cast<uint4*>(c);
#pragma unroll
      for (int j = 0; j < 4; j++) d[j] = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
    } else {
#pragma unroll
      for (int j = 0; j < 32; j++)
        if (n0 + j < p.N) c[j] = __float2half_rn(__uint_as_float(r[j]));
    }
  } else {
    float* c = reinterpret_cast<float*>(p.C) + m * p.N + n0;
    if (n0 + 32 <= p.N && (p.N & 3) == 0) {
      float4* d = reinterpret_cast<float4*>(c);
      float4 o[8];
      if (is_resid(EPI)) {
#pragma unroll
        for (int j = 0; j < 8; j++) o[j] = d[j];  // all loads in flight before the first store
      }
#pragma unroll
      for (int j = 0; j < 8; j++) {
        float4 v = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]), __uint_as_float(r[4 * j + 2]),
                               __uint_as_float(r[4 * j + 3]));
        if (is_resid(EPI)) {
          v.x += o[j].x;
          v.y += o[j].y;
          v.z += o[j].z;
          v.w += o[j].w;
        }
        __stcs(d + j, v);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; j++)
        if (n0 + j < p.N) c[j] = (is_resid(EPI) ? c[j] : 0.f) + __uint_as_float(r[j]);
    }
  }
}

template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(EpiShape<EPI>::kThreads, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tma_a, const __grid_constant__ CUtensorMap tma_b, Params p) {
  constexpr int STAGES = EpiShape<EPI>::kStages, KSUB = EpiShape<EPI>::kSub;
  constexpr uint32_t A_BYTES = KSUB * A_SUB, STAGE_BYTES = KSUB * (A_SUB + B_SUB);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 4);
  float* staging = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES + 256);
  const uint32_t smem_base = smem_u32(smem);
  auto sA = [&](int s) { return smem_base + (uint32_t)s * STAGE_BYTES; };
  auto sB = [&](int s) { return smem_base + (uint32_t)s * STAGE_BYTES + A_BYTES; };
  auto full = [&](int s) { return smem_u32(bars + s); };
  auto empty = [&](int s) { return smem_u32(bars + STAGES + s); };
  auto tfull = [&](int a) { return smem_u32(bars + 2 * STAGES + a); };
  auto tempty = [&](int a) { return smem_u32(bars + 2 * STAGES + 2 + a); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t rank;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const bool leader = rank == 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; s++) {
      mbar_init(full(s), 1);   // the leader's: its expect_tx arrival plus both CTAs' bytes
      mbar_init(empty(s), 1);  // the leader's multicast commit
    }
    for (int a = 0; a < 2; a++) {
      mbar_init(tfull(a), 1);                           // the leader's multicast commit
      mbar_init(tempty(a), 2 * 32 * EpiShape<EPI>::kWarps);  // the leader's: both CTAs' epilogues
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    // one warp of each CTA of the pair allocates together (the same columns in both)
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_tiles = p.tiles_m * p.tiles_n;
  const int cid = (int)(blockIdx.x >> 1), ncl = (int)(gridDim.x >> 1);

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    // the weight operand B is re-read by every group of M-blocks: keep it in L2 ahead of the
    // streamed activations
    uint64_t keep_b;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep_b));
    uint32_t g = 0;
    bool ok = true;
    const int a_row = (int)rank * BM, b_row = (int)rank * (BN / 2);
    for (int t = cid; t < n_tiles && ok; t += ncl) {
      int mb, nb;
      tile_coords(t, p, mb, nb);
      for (int kb = 0; kb < p.num_kb; ++kb, ++g) {
        const int s = (int)(g % STAGES);
        const uint32_t ph = (g / STAGES) & 1u;
        ok = __all_sync(0xffffffffu, mbar_wait(empty(s), ph ^ 1u, p.err));
        if (!ok) break;
        if (lane == 0) {
          const uint32_t lf = cluster_addr(full(s), 0);
          if (leader) mbar_expect_tx(full(s), 2 * STAGE_BYTES);
#pragma unroll
          for (int u = 0; u < KSUB; u++) {
            const int kx = (kb * KSUB + u) * BK;
            tma_load_pair(sA(s) + u * A_SUB, &tma_a, lf, kx, mb * TM + a_row);
            if (p.keep_b) tma_load_pair_hint(sB(s) + u * B_SUB, &tma_b, lf, kx, nb * BN + b_row, keep_b);
            else tma_load_pair(sB(s) + u * B_SUB, &tma_b, lf, kx, nb * BN + b_row);
          }
        }
        __syncwarp();
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (the leader CTA) ----------------
    uint32_t g = 0;
    int i = 0;
    bool ok = leader;
    for (int t = cid; t < n_tiles && ok; t += ncl, ++i) {
      const int a = i & 1;
      const uint32_t aph = (uint32_t)(i >> 1) & 1u;
      ok = __all_sync(0xffffffffu, mbar_wait(tempty(a), aph ^ 1u, p.err));
      if (!ok) break;
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(a * BN);
      for (int kb = 0; kb < p.num_kb; ++kb, ++g) {
        const int s = (int)(g % STAGES);
        const uint32_t ph = (g / STAGES) & 1u;
        ok = __all_sync(0xffffffffu, mbar_wait(full(s), ph, p.err));
        if (!ok) break;
        tc_fence_after();
        if (lane == 0) {
#pragma unroll
          for (int u = 0; u < KSUB; ++u) {
            const uint64_t da = sw128_desc(sA(s) + u * A_SUB), db = sw128_desc(sB(s) + u * B_SUB);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)
              tc_mma(d, da + (uint64_t)(2 * k), db + (uint64_t)(2 * k), (kb > 0 || u > 0 || k > 0) ? 1u : 0u);
          }
          tc_commit_pair(empty(s));
        }
        __syncwarp();
      }
      if (lane == 0) tc_commit_pair(tfull(a));
      __syncwarp();
    }
  } else {
    // ---------------- epilogue (warps 2 ..) ----------------
    constexpr int NH = EpiShape<EPI>::kWarps / 4;  // column parts of a tile
    constexpr int HN = BN / NH;
    const int q = warp & 3;            // TMEM lanes 32q .. 32q+31
    const int hw = (warp - 2) >> 2;    // tile columns [HN hw, HN hw + HN)
    float* stg = staging + (warp - 2) * (NH == 2 ? 32 * 32 : 32 * 36);
    int i = 0;
    const uint32_t tempty_leader0 = cluster_addr(tempty(0), 0), tempty_leader1 = cluster_addr(tempty(1), 0);
    for (int t = cid; t < n_tiles; t += ncl, ++i) {
      int mb, nb;
      tile_coords(t, p, mb, nb);
      const int a = i & 1;
      const uint32_t aph = (uint32_t)(i >> 1) & 1u;
      const int64_t mrow0 = (int64_t)mb * TM + (int64_t)rank * BM;  // this CTA's first tile row
      const int64_t m = mrow0 + q * 32 + lane;
      const int64_t ncol0 = (int64_t)nb * BN + hw * HN;  // first output column of this half
      // pull this half-tile's residual rows into L2 while its accumulator is still being built
      if (is_resid(EPI) && (p.N & 31) == 0) prefetch_residual(p, m, ncol0, HN);
      const float rs = row_scale(p, m);
      if (!__all_sync(0xffffffffu, mbar_wait(tfull(a), aph, p.err))) break;
      tc_fence_after();
      const uint32_t tacc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(a * BN);  // tile column 0
      const uint32_t tbase = tacc + (uint32_t)(hw * HN);
      if (EPI == kQKVRope) {
        // one head at a time (a half holds HN / hd whole heads): halves [0, hd/2) and [hd/2, hd)
        // rotate pairwise by pos * theta_i
        const int hd = p.rope_hd, hh = hd / 2;
        const int64_t pos = p.rope_pos0 + m % p.rope_pos_mod;
        const float2* cs = p.rope_cs + pos * hh;
#pragma unroll 1
        for (int c = 0; c < hh / 32; ++c) {
          float ct[32], st[32];
          const bool any_rot = ncol0 < p.rope_cols && m < p.M;
          if (any_rot) {
            const float4* c4 = reinterpret_cast<const float4*>(cs + c * 32);
#pragma unroll
            for (int j = 0; j < 16; j++) {
              const float4 t = __ldg(c4 + j);
              ct[2 * j] = t.x;
              st[2 * j] = t.y;
              ct[2 * j + 1] = t.z;
              st[2 * j + 1] = t.w;
            }
          }
#pragma unroll 1
          for (int hs = 0; hs < HN / hd; ++hs) {
            const int64_t col0 = ncol0 + hs * hd;
            const bool rot = col0 < p.rope_cols;
            uint32_t a[32], b[32];
            tmem_ld32(tbase + (uint32_t)(hs * hd + c * 32), a);
            tmem_ld32(tbase + (uint32_t)(hs * hd + hh + c * 32), b);
            if (m < p.M && col0 < p.N) {
              if (rot) {
#pragma unroll
                for (int j = 0; j < 32; j++) {
                  const float x = __uint_as_float(a[j]) * rs, y = __uint_as_float(b[j]) * rs;
                  a[j] = __float_as_uint(x * ct[j] - y * st[j]);
                  b[j] = __float_as_uint(x * st[j] + y * ct[j]);
                }
              } else if (p.row_ss) {
#pragma unroll
                for (int j = 0; j < 32; j++) {
                  a[j] = __float_as_uint(__uint_as_float(a[j]) * rs);
                  b[j] = __float_as_uint(__uint_as_float(b[j]) * rs);
                }
              }
              store_chunk<kStore>(p, m, col0 + c * 32, a);
              store_chunk<kStore>(p, m, col0 + hh + c * 32, b);
            }
          }
        }
      } else if (EPI == kSwiGLU) {
        // columns [0, 128) of the tile are gate, [128, 256) the matching up columns; this warp
        // writes output chunks [4 hw / NH, 4 (hw + 1) / NH) (32 columns each)
#pragma unroll 1
        for (int c = 4 * hw / NH; c < 4 * (hw + 1) / NH; ++c) {
          uint32_t g[32], u[32];
          tmem_ld32(tacc + (uint32_t)(c * 32), g);
          tmem_ld32(tacc + (uint32_t)(BN / 2 + c * 32), u);
          if (m < p.M) {
            const int64_t half_n = p.N / 2;
            __half* dst = reinterpret_cast<__half*>(p.C) + m * half_n + (int64_t)nb * (BN / 2) + c * 32;
            uint32_t w[16];
#pragma unroll
            for (int j = 0; j < 16; j++) {
              const float g0 = __uint_as_float(g[2 * j]) * rs, g1 = __uint_as_float(g[2 * j + 1]) * rs;
              const float a0 = g0 / (1.f + expf(-g0)) * (__uint_as_float(u[2 * j]) * rs);
              const float a1 = g1 / (1.f + expf(-g1)) * (__uint_as_float(u[2 * j + 1]) * rs);
              __half2 h = __floats2half2_rn(a0, a1);
              w[j] = *reinterpret_cast<uint32_t*>(&h);
            }
            uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
            for (int j = 0; j < 4; j++) d4[j] = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
          }
        }
      } else if ((is_resid(EPI) || EPI == kStoreF32) && (p.N & 31) == 0) {
        // fp32 output through a shared-memory transpose: the warp's 32 rows x 32 columns go in one
        // row per thread and come out as 8 lanes per row, so each global access covers 4 full rows
        // of 128 B. The residual forms add the stored x; with xh set they also write fp16(x), and
        // ss_out[row * tiles_n * NH + nb * NH + hw] receives the row's sum of squares over this
        // warp's columns of the tile: all of them with 4 epilogue warps, half with 8 (fixed order:
        // per lane over chunks, then a butterfly over the row's 8 lanes).
        const int cr = lane >> 3, sl = lane & 7, cc = sl * 4;
        const int64_t row0 = mrow0 + q * 32;
        float rmax = -INFINITY;  // kStoreF32: this thread's row (m) over its columns
        float ssl[8];
#pragma unroll
        for (int k = 0; k < 8; k++) ssl[k] = 0.f;
#pragma unroll 1
        for (int c = 0; c < HN / 32; ++c) {
          const int64_t n0 = ncol0 + c * 32;
          if (n0 >= p.N) break;
          uint32_t r[32];
          tmem_ld32(tbase + (uint32_t)(c * 32), r);
          if (p.row_ss) {
#pragma unroll
            for (int j = 0; j < 32; j++) r[j] = __float_as_uint(__uint_as_float(r[j]) * rs);
          }
          if (EPI == kStoreF32 && p.row_max) {
#pragma unroll
            for (int j = 0; j < 32; j += 2) rmax = fmaxf(rmax, fmaxf(__uint_as_float(r[j]), __uint_as_float(r[j + 1])));
          }
#pragma unroll
          for (int j = 0; j < 8; j++)
            *reinterpret_cast<float4*>(stg + stg_off<NH>(lane, j)) =
                make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]), __uint_as_float(r[4 * j + 2]),
                            __uint_as_float(r[4 * j + 3]));
          __syncwarp();
          float* cbase = reinterpret_cast<float*>(p.C) + n0 + cc;
          float4 o[8];
          if (is_resid(EPI)) {
#pragma unroll
            for (int k = 0; k < 8; k++) {
              const int64_t gm = row0 + 4 * k + cr;
              o[k] = gm < p.M ? __ldcs(reinterpret_cast<const float4*>(cbase + gm * p.N))
                              : make_float4(0.f, 0.f, 0.f, 0.f);
            }
          }
#pragma unroll
          for (int k = 0; k < 8; k++) {
            const int rr = 4 * k + cr;
            const int64_t gm = row0 + rr;
            const float4 acc = *reinterpret_cast<const float4*>(stg + stg_off<NH>(rr, sl));
            float4 v = acc;
            if (is_resid(EPI)) {
              v.x = o[k].x + acc.x;
              v.y = o[k].y + acc.y;
              v.z = o[k].z + acc.z;
              v.w = o[k].w + acc.w;
            }
            if (gm < p.M) {
              __stcs(reinterpret_cast<float4*>(cbase + gm * p.N), v);
              if (is_resid(EPI) && p.xh) {
                __half2 h0 = __floats2half2_rn(v.x, v.y), h1 = __floats2half2_rn(v.z, v.w);
                __stcs(reinterpret_cast<uint2*>(p.xh + gm * p.N + n0 + cc),
                       make_uint2(*reinterpret_cast<uint32_t*>(&h0), *reinterpret_cast<uint32_t*>(&h1)));
              }
            }
            ssl[k] += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
          }
          __syncwarp();
        }
        if (EPI == kStoreF32 && p.row_max && m < p.M && rmax != -INFINITY)
          atomicMax(p.row_max + m, float_key(__float_as_uint(rmax)));
        if (is_resid(EPI) && p.xh) {
#pragma unroll
          for (int k = 0; k < 8; k++) {
            float v = ssl[k];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            const int64_t gm = row0 + 4 * k + cr;
            if ((lane & 7) == 0 && gm < p.M) p.ss_out[gm * (p.tiles_n * NH) + nb * NH + hw] = v;
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < HN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tbase + (uint32_t)(c * 32), r);
          const int64_t n0 = ncol0 + c * 32;
          if (p.row_ss) {
#pragma unroll
            for (int j = 0; j < 32; j++) r[j] = __float_as_uint(__uint_as_float(r[j]) * rs);
          }
          if (m < p.M && n0 < p.N) store_chunk<EPI>(p, m, n0, r);
        }
      }
      tc_fence_before();
      mbar_arrive_cluster(a ? tempty_leader1 : tempty_leader0);
    }
  }
  // neither CTA leaves (or frees its tensor memory) while the pair's MMAs may still use it
  tc_fence_before();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
  }
}

// ---------------- host side ----------------
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static std::once_flag g_once;
static int g_num_sms = 0;
static int g_max_clusters[6] = {0, 0, 0, 0, 0, 0};  // co-resident CTA pairs, per epilogue kind

template <int EPI>
static void setup_kernel() {
  cudaFuncSetAttribute(k_gemm_tc<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes<EPI>());
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::max(2, g_num_sms & ~1), 1, 1);
  cfg.blockDim = dim3(EpiShape<EPI>::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes<EPI>();
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k_gemm_tc<EPI>, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = g_num_sms / 2;
  }
  g_max_clusters[EPI] = std::max(1, n);
}

static void init_once() {
  cudaDriverEntryPointQueryResult q;
  void* fn = nullptr;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10) g_encode = nullptr;  // tcgen05 path only on Blackwell-class devices
  if (!g_encode) return;
  setup_kernel<kStore>();
  setup_kernel<kAddResidual>();
  setup_kernel<kAddResidualWide>();
  setup_kernel<kStoreF32>();
  setup_kernel<kSwiGLU>();
  setup_kernel<kQKVRope>();
}

static bool make_map(CUtensorMap* map, const void* ptr, uint64_t k, uint64_t rows, uint32_t box_rows) {
  cuuint64_t dims[2] = {k, rows};
  cuuint64_t strides[1] = {k * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace tc

bool tc_gemm_supported(int64_t M, int64_t N, int64_t K, int epi) {
  std::call_once(tc::g_once, tc::init_once);
  if (epi == kSwiGLU && N % tc::BN != 0) return false;
  if (epi == kQKVRope && N % 64 != 0) return false;
  return tc::g_encode != nullptr && M > 0 && N > 0 && K > 0 && K % 8 == 0 && M < (1ll << 31) && N < (1ll << 31);
}

void launch_gemm_tc(const void* A, const void* B, void* C, int64_t M, int64_t N, int64_t K, int epi, uint32_t* err,
                    cudaStream_t s, const RopeArgs* rope, const NormArgs* norm) {
  using namespace tc;
  std::call_once(g_once, init_once);
  CUtensorMap ma, mb;
  if (!make_map(&ma, A, (uint64_t)K, (uint64_t)M, BM) || !make_map(&mb, B, (uint64_t)K, (uint64_t)N, BN / 2)) {
    set_thread_error("cuTensorMapEncodeTiled failed");
    return;
  }
  Params p;
  p.C = C;
  p.M = M;
  p.N = N;
  p.K = K;
  p.tiles_m = (int)((M + TM - 1) / TM);
  p.tiles_n = (int)((N + BN - 1) / BN);
  const int ksub = epi == kStoreF32 ? EpiShape<kStoreF32>::kSub : EpiShape<kStore>::kSub;
  p.num_kb = (int)((K + ksub * BK - 1) / (ksub * BK));  // ring stages along K
  p.keep_b = N * K * 2 <= kKeepBBytes ? 1 : 0;
  // wide GEMMs (many N tiles) sweep an L2-resident weight fewer times with 32 pair tiles per
  // group; narrow ones keep 8 so that a wave of 76 pairs spans whole groups; a streamed weight
  // takes 16
  p.group_m = p.keep_b ? (p.tiles_n < 16 ? 8 : 32) : 16;
  p.err = err;
  p.rope_cs = rope ? rope->cs : nullptr;
  p.rope_cols = rope ? rope->cols : 0;
  p.rope_hd = rope ? rope->hd : 64;
  p.rope_pos_mod = rope ? rope->pos_mod : 1;
  p.rope_pos0 = rope ? rope->pos0 : 0;
  p.row_ss = norm ? norm->row_ss : nullptr;
  p.ss_parts = norm ? norm->parts : 0;
  p.ss_inv_d = norm ? norm->inv_d : 0.f;
  p.ss_eps = norm ? norm->eps : 0.f;
  p.xh = norm ? norm->xh : nullptr;
  p.ss_out = norm ? norm->ss_out : nullptr;
  p.row_max = norm ? norm->row_max : nullptr;
  const int tiles = p.tiles_m * p.tiles_n;
  const int grid = 2 * std::max(1, std::min(tiles, g_max_clusters[epi]));  // CTA pairs
  note_launch();
  if (epi == kStore) k_gemm_tc<kStore><<<grid, EpiShape<kStore>::kThreads, smem_bytes<kStore>(), s>>>(ma, mb, p);
  else if (epi == kAddResidual)
    k_gemm_tc<kAddResidual><<<grid, EpiShape<kAddResidual>::kThreads, smem_bytes<kAddResidual>(), s>>>(ma, mb, p);
  else if (epi == kAddResidualWide)
    k_gemm_tc<kAddResidualWide>
        <<<grid, EpiShape<kAddResidualWide>::kThreads, smem_bytes<kAddResidualWide>(), s>>>(ma, mb, p);
  else if (epi == kStoreF32) k_gemm_tc<kStoreF32><<<grid, EpiShape<kStoreF32>::kThreads, smem_bytes<kStoreF32>(), s>>>(ma, mb, p);
  else if (epi == kSwiGLU) k_gemm_tc<kSwiGLU><<<grid, EpiShape<kSwiGLU>::kThreads, smem_bytes<kSwiGLU>(), s>>>(ma, mb, p);
  else k_gemm_tc<kQKVRope><<<grid, EpiShape<kQKVRope>::kThreads, smem_bytes<kQKVRope>(), s>>>(ma, mb, p);
}

}  // namespace lmgc
