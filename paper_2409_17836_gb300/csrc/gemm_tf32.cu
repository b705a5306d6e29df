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
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "lmgc_internal.cuh"

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
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, uint32_t* err) {
  if (mbar_try(a, parity)) return true;
  uint64_t t0, t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (uint32_t i = 1; i < (1u << 28); ++i) {
    if (mbar_try(a, parity)) return true;
    if ((i & 127) == 0) {
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
      if (t - t0 > 2000000000ull) break;
    }
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
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(
          d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// K-major operand, 128-byte swizzle: 8-row groups 1024 B apart (SBO), LBO unused; an 8-wide TF32
// K slice starts 32 bytes further into each 128-byte row
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
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

// x -> (hi, lo) in place: hi (x with its low 13 bits cleared) over x, lo = x - hi at lo_off
// bytes further on; n16 16-byte units shared by the 128 splitting threads
__device__ __forceinline__ void split_tile(uint8_t* base, uint32_t lo_off, int n16, int t) {
  for (int i = t; i < n16; i += 128) {
    float4* x = reinterpret_cast<float4*>(base) + i;
    float4* y = reinterpret_cast<float4*>(base + lo_off) + i;
    const float4 v = *x;
    float4 h, l;
    h.x = __uint_as_float(__float_as_uint(v.x) & 0xFFFFE000u);
    h.y = __uint_as_float(__float_as_uint(v.y) & 0xFFFFE000u);
    h.z = __uint_as_float(__float_as_uint(v.z) & 0xFFFFE000u);
    h.w = __uint_as_float(__float_as_uint(v.w) & 0xFFFFE000u);
    l.x = __fsub_rn(v.x, h.x);
    l.y = __fsub_rn(v.y, h.y);
    l.z = __fsub_rn(v.z, h.z);
    l.w = __fsub_rn(v.w, h.w);
    *x = h;
    *y = l;
  }
}

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
  if (major != 10) g_encode = nullptr;  // tcgen05 path only on Blackwell-class devices
  if (!g_encode) return;
  cudaFuncSetAttribute(k_gemm_tf32x3<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<128>::SMEM);
  cudaFuncSetAttribute(k_gemm_tf32x3<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<32>::SMEM);
}

static bool make_map(CUtensorMap* map, const void* ptr, uint64_t k, uint64_t rows, uint32_t box_rows) {
  cuuint64_t dims[2] = {k, rows};
  cuuint64_t strides[1] = {k * 4};
  cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
