// gemm_tf32.cu -- the dense contractions of an fp32 model (Eq. 2's linear layers and vocabulary
// projection, C = A . B^T with A [M][K], B [N][K] row-major fp32) on the 5th-generation tensor
// cores in three-pass TF32 form.
//
// A tcgen05 MMA of kind::tf32 reads only the top 19 bits of each fp32 operand (sign, exponent,
// 10 mantissa bits). Each operand x is split into hi = x with its low 13 bits cleared and lo =
// x - hi (exact in fp32, |lo| < 2^-10 |x|), and C accumulates lo_A hi_B + hi_A lo_B + hi_A hi_B
// in fp32 in tensor memory: the dropped lo_A lo_B term and lo's own truncation to 10 mantissa
// bits are each below 2^-20 |a b|, so the result is within about 2^-18 sum_k |a_k b_k| of the
// exact product, the 1e-3 bound on fp32 logits with margin to spare.
//
// One CTA per 128 x BN tile of C (BN = 128, or 32 for N <= 32); 192 threads:
//   warp 0      TMA: the fp32 A (128 x 32) and B (BN x 32) tiles of each K step into a 3-stage ring
//   warp 1      TMEM allocation; one lane issues the three MMA streams per 8-wide K slice and
//               commits each stage back to the producer
//   warps 2-5   split each landed stage in place (hi over x, lo beside it; the 128-byte swizzle
//               only permutes positions, and the split is elementwise), then, after the last K
//               step, the epilogue: TMEM lane quarter w % 4, one row of C per thread
// Every mbarrier wait is bounded (~2 s), after which kErrLimit is recorded and the loops end.
// Rows are independent (no split-K, a row's K order fixed), so a decode step's rows match the
// prefill's bit for bit.
#include "tf32_common.cuh"

namespace lmgc {
namespace tf32 {

constexpr int BM = 128, BK = 32, kStages = 3, kThreads = 192;

template <int BN>
struct Cfg {
  static constexpr uint32_t A_BYTES = BM * BK * 4;  // 16 KiB: 128 rows of 128 bytes
  static constexpr uint32_t B_BYTES = BN * BK * 4;
  // stage: A (hi after the split) | A lo | B (hi) | B lo, each 1024-byte aligned
  static constexpr uint32_t STAGE = 2 * A_BYTES + 2 * B_BYTES;
  static constexpr uint32_t TMEM_COLS = BN;  // 32 or 128 (powers of two, at least 32)
  static constexpr size_t SMEM = kStages * STAGE + 1024 + 256;
  // instruction descriptor, kind::tf32: D fp32 (bits 4-5 = 1), A and B TF32 (bits 7-9, 10-12 =
  // 2), both K-major, N >> 3 at bit 17, M >> 4 at bit 24
  static constexpr uint32_t IDESC =
      (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
};

struct Params {
  float* C;
  int64_t M, N, K;
  int epi;  // kStore / kStoreF32: C = A B^T; kAddResidual: C += A B^T
  uint32_t* err;
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_tf32x3(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, Params p) {
  using G = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * G::STAGE);
  // barriers: 0-2 stage landed (TMA) | 3-5 stage split (128 arrivals) | 6-8 stage read by the
  // MMAs (commit) | 9 all MMAs done (commit)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 12);
  auto b_full = [&](int s) { return smem_u32(bars + s); };
  auto b_split = [&](int s) { return smem_u32(bars + 3 + s); };
  auto b_empty = [&](int s) { return smem_u32(bars + 6 + s); };
  const uint32_t b_done = smem_u32(bars + 9);
  auto stage = [&](int s) { return smem + (size_t)s * G::STAGE; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
  const int nk = (int)((p.K + BK - 1) / BK);

  if (threadIdx.x == 0) {
    for (int i = 0; i < 10; i++) mbar_init(smem_u32(bars + i), (i >= 3 && i <= 5) ? 128 : 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(G::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    for (int kt = 0; kt < nk; kt++) {
      const int s = kt % kStages;
      // the stage is free once the MMAs of K step kt - kStages have read it (this warp saw its
      // previous release; the next needs step kt, which needs this load)
      if (kt >= kStages &&
          !__all_sync(0xffffffffu, mbar_wait(b_empty(s), (uint32_t)((kt - kStages) / kStages) & 1u, p.err)))
        break;
      if (lane == 0) {
        mbar_expect_tx(b_full(s), G::A_BYTES + G::B_BYTES);
        tma_load_2d(smem_u32(stage(s)), &ta, b_full(s), kt * BK, (int)m0);
        tma_load_2d(smem_u32(stage(s) + 2 * G::A_BYTES), &tb, b_full(s), kt * BK, (int)n0);
      }
      __syncwarp();
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: lo_A hi_B, hi_A lo_B, hi_A hi_B per 8-wide K slice ----------------
    bool ok = true;
    for (int kt = 0; kt < nk && ok; kt++) {
      const int s = kt % kStages;
      // split(kt) (its previous phase, split(kt - kStages), was seen here; the next needs a load
      // that waits for this step's release)
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(b_split(s), (uint32_t)(kt / kStages) & 1u, p.err)))) break;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t a_hi = smem_u32(stage(s)), a_lo = a_hi + G::A_BYTES;
        const uint32_t b_hi = a_hi + 2 * G::A_BYTES, b_lo = b_hi + G::B_BYTES;
#pragma unroll
        for (int k = 0; k < BK / 8; k++) {
          const uint32_t o = 32u * k;
          tc_mma(tmem, desc_kmajor(a_lo + o), desc_kmajor(b_hi + o), G::IDESC, (kt > 0 || k > 0) ? 1u : 0u);
          tc_mma(tmem, desc_kmajor(a_hi + o), desc_kmajor(b_lo + o), G::IDESC, 1u);
          tc_mma(tmem, desc_kmajor(a_hi + o), desc_kmajor(b_hi + o), G::IDESC, 1u);
        }
        tc_commit(b_empty(s));
        if (kt == nk - 1) tc_commit(b_done);
      }
      __syncwarp();
    }
  } else {
    // ---------------- split, then epilogue (warps 2-5) ----------------
    const int t = threadIdx.x - 64;
    bool ok = true;
    for (int kt = 0; kt < nk && ok; kt++) {
      const int s = kt % kStages;
      // the load of step kt (its previous phase was seen here; the next needs the stage's release,
      // which needs this split)
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(b_full(s), (uint32_t)(kt / kStages) & 1u, p.err)))) break;
      uint8_t* st = stage(s);
      split_tile(st, G::A_BYTES, (int)(G::A_BYTES / 16), t);
      split_tile(st + 2 * G::A_BYTES, G::B_BYTES, (int)(G::B_BYTES / 16), t);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the MMAs read these writes
      mbar_arrive(b_split(s));
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(b_done, 0u, p.err));
    if (ok) {
      tc_fence_after();
      const int q = warp & 3;  // TMEM lane quarter of this warp
      const int64_t m = m0 + 32 * q + lane;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c0, r);
        if (m >= p.M) continue;
        float* crow = p.C + m * p.N + n0 + c0;
        const int64_t nv = p.N - (n0 + c0);  // valid columns from c0
        if (nv >= 32 && (p.N & 3) == 0) {
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            float4 v = make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]), __uint_as_float(r[j + 2]),
                                   __uint_as_float(r[j + 3]));
            float4* dst = reinterpret_cast<float4*>(crow + j);
            if (p.epi == kAddResidual) {
              const float4 o = *dst;
              v.x += o.x;
              v.y += o.y;
              v.z += o.z;
              v.w += o.w;
            }
            *dst = v;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; j++) {
            if (j >= nv) break;
            const float v = __uint_as_float(r[j]);
            crow[j] = p.epi == kAddResidual ? crow[j] + v : v;
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(G::TMEM_COLS) : "memory");
  }
}

static std::once_flag g_once;
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn_enc = nullptr;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn_enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    int dev = 0, major = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (major != 10) fn_enc = nullptr;  // tcgen05 path only on Blackwell-class devices
  });
  return fn_enc;
}

bool make_map_f32(CUtensorMap* map, const void* ptr, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 4};
  cuuint32_t box[2] = {32u, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(ptr), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static void init_once() {
  g_encode = encoder();
  if (!g_encode) return;
  cudaFuncSetAttribute(k_gemm_tf32x3<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<128>::SMEM);
  cudaFuncSetAttribute(k_gemm_tf32x3<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<32>::SMEM);
}

static bool make_map(CUtensorMap* map, const void* ptr, uint64_t k, uint64_t rows, uint32_t box_rows) {
  return make_map_f32(map, ptr, k, rows, box_rows);
}
}  // namespace tf32

bool tf32_gemm_supported(int64_t M, int64_t N, int64_t K) {
  std::call_once(tf32::g_once, tf32::init_once);
  return tf32::g_encode != nullptr && M > 0 && N > 0 && K > 0 && K % 4 == 0 && M < (1ll << 31) &&
         N < (1ll << 31);
}

void launch_gemm_tf32(const float* A, const float* B, float* C, int64_t M, int64_t N, int64_t K, int epi,
                      uint32_t* err, cudaStream_t s) {
  using namespace tf32;
  std::call_once(g_once, init_once);
  if (M <= 0 || N <= 0) return;
  const bool narrow = N <= 32;
  CUtensorMap ma, mb;
  if (!g_encode || !make_map(&ma, A, (uint64_t)K, (uint64_t)M, BM) ||
      !make_map(&mb, B, (uint64_t)K, (uint64_t)N, narrow ? 32u : 128u)) {
    set_thread_error("cuTensorMapEncodeTiled failed (tf32 gemm)");
    return;
  }
  Params p;
  p.C = C;
  p.M = M;
  p.N = N;
  p.K = K;
  p.epi = epi == kAddResidualWide ? (int)kAddResidual : epi;
  p.err = err;
  note_launch();
  if (narrow) {
    dim3 grid(1u, (unsigned)((M + BM - 1) / BM));
    k_gemm_tf32x3<32><<<grid, kThreads, Cfg<32>::SMEM, s>>>(ma, mb, p);
  } else {
    dim3 grid((unsigned)((N + 127) / 128), (unsigned)((M + BM - 1) / BM));
    k_gemm_tf32x3<128><<<grid, kThreads, Cfg<128>::SMEM, s>>>(ma, mb, p);
  }
}

}  // namespace lmgc
