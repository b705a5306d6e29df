// coder.cu -- the arithmetic coder (Sec. 3 "Arithmetic coding") in exact integer form, one
// independent stream per window (Sec. 4 "Compression": each window is coded from its own BOS).
//
// Per stream: R = 2^62, L = 0, B = 0; per token (s = start, f = freq, T = 2^P):
//   r = R >> P;  L += r*s;  R = r*f;  k = max(0, 62 - bitlen(R));  R <<= k;  L <<= k;  B += k
// and the code is the top B + 2 bits of v = ceil(L / 2^60) * 2^60 (v lies in [L, L + R) because
// R >= 2^61), most significant bit first.
//
// Form computed here (the same integers, no shift of L). R depends only on the freq sequence, and
// only r = R >> P is kept: after R = r f and the shift by k, the next r is (r f) >> (P - k), with
// k = clz(r f) - 2 over 64 bits (0 for r f = 2^62). In stream coordinates (bit j of the code has
// weight 2^-(j+1)) token i's addend r s occupies bits [B_i, B_i + 62), B_i being the shift total
// before it, so L is the sum of the addends at their positions. A thread keeps stream bits
// [32 w, 32 w + 96) in three registers a0:a1:a2 and adds each addend at offset off = B - 32 w,
// which stays in [3, 34] between tokens (sh = 34 - off is a funnel-shift count below 32). Word a0
// is complete when off reaches 35: it moves to a fourth register am1, the window moves one word
// on, and the word am1 held leaves. A carry out of a0 goes into am1 within the same add; one out
// of am1 (only when am1 is all ones) increments the completed words before it (never beyond
// word 0: L + R stays below 2^(B+62)).
//
// Per token: two 32x32->64 multiply-adds per product, three funnel shifts, a four-word add with
// carry, a count of leading zeros and a handful of selects (the step is inline PTX so that each
// operation is one instruction). Completed words go to a per-thread ring in shared memory and
// leave for the stream's slot in 16-byte chunks, at most two per 8 tokens: scattered 4-byte
// stores from 32 lanes to 32 slots would cost one memory transaction each. The tiled coder
// interleaves the slots of a warp's 32 windows chunk by chunk (chunk c of window w at
// (c * 32 + w % 32) * 16 bytes into the block's table), so that the chunks the 32 streams flush
// at about the same point of their codes share memory lines.
//
// Layout: one stream per thread, 32 windows per warp. Pairs come from window tiles (the encode
// path; a warp's 8 tokens are one contiguous kilobyte per array, staged through shared memory by
// asynchronous copies) or from start[w*stride_win + i*stride_pos] (lmgc_range_encode's general layout,
// loaded 8 tokens ahead).
// Slot words are stored in native byte order; the pack step writes the bytes most significant
// first.
#include <algorithm>
#include <mutex>
#include <string>

#include "lmgc_internal.cuh"

namespace lmgc {

// ceil((W P + 2) / 32) + 1 words, rounded up to 16 bytes (whole 16-byte chunks)
size_t slot_bytes(size_t win_tokens, int P) {
  size_t bits = win_tokens * (size_t)P + 2;
  size_t words = (bits + 31) / 32 + 1;
  return ((words * 4 + 15) / 16) * 16;
}

constexpr int kRingWords = 16;   // completed words not yet written (at most 4 + 8 between flushes)
constexpr int kRingStride = 20;  // words per thread in shared memory: 16-byte aligned, few bank conflicts
constexpr int kCoderThreads = 128;

template <bool ILV>
struct Stream {
  uint32_t rlo, rhi;   // r = R >> P
  uint32_t a0, a1, a2; // stream bits [32 w, 32 w + 96)
  uint32_t am1;        // word w - 1, the last completed one (a carry out of a0 lands here)
  uint32_t nz;         // OR of the words below word 0 as they completed (checked form; zero for valid input)
  int32_t sh;          // 34 - (B - 32 w), in [0, 31] between tokens
  int32_t w;           // word index of a0 (-1 before the first word completes)
  int32_t fw;          // words [0, fw) are in the slot, [fw, w - 1) only in the ring
  uint32_t chk;        // OR of s | (f - 1) | (s + f - 1) over the tokens: >= T iff a pair was invalid
  uint32_t max_words;
  uint32_t* slot;       // the window's slot, or (ILV) the warp's table of 32 interleaved slots
  uint32_t lane;        // ILV: this window's column of the table
  uint32_t ring;        // shared-memory address of this thread's ring (kRingWords words)
  bool overflow;

  // ring words through shared-state-space instructions (a generic pointer would make every
  // read of the ring wait like a global load)
  __device__ __forceinline__ uint32_t ring_ld(int32_t i) const {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(ring + 4u * (uint32_t)(i & (kRingWords - 1))) : "memory");
    return v;
  }
  __device__ __forceinline__ void ring_st(int32_t i, uint32_t v) const {
    asm volatile("st.shared.u32 [%0], %1;" ::"r"(ring + 4u * (uint32_t)(i & (kRingWords - 1))), "r"(v) : "memory");
  }
  // word i of the code: slot[i], or (ILV) 16-byte chunk i / 4 of the window's column, so that
  // the chunks the 32 windows of a warp write at about the same point of their codes lie side by
  // side (a warp's chunk stores then touch few memory lines instead of 32)
  __device__ __forceinline__ uint32_t* word(int32_t i) const {
    return ILV ? slot + ((size_t)(uint32_t)(i >> 2) * 32u + lane) * 4u + (uint32_t)(i & 3) : slot + i;
  }
  __device__ __forceinline__ void init(int P, uint32_t* sl, uint32_t mw, uint32_t* rg, uint32_t ln = 0) {
    lane = ln;
    const uint64_t r0 = 1ull << (62 - P);  // R = 2^62
    rlo = (uint32_t)r0;
    rhi = (uint32_t)(r0 >> 32);
    a0 = a1 = a2 = am1 = nz = 0u;
    sh = 2;  // B = 0 at w = -1: off = 32
    w = -1;
    fw = 0;
    chk = 0u;
    max_words = mw;
    slot = sl;
    ring = (uint32_t)__cvta_generic_to_shared(rg);
    overflow = false;
  }
  // +1 into the completed words before am1 (ring or slot); a carry past word 0 cannot happen for
  // valid input and is reported
  __device__ __forceinline__ void carry() {
    for (int32_t i = w - 2; i >= 0; --i) {
      uint32_t v;
      if (i >= fw) {
        v = ring_ld(i) + 1u;
        ring_st(i, v);
      } else {
        if ((uint32_t)i >= max_words) break;
        v = *word(i) + 1u;
        *word(i) = v;
      }
      if (v != 0u) return;
    }
    overflow = true;
  }
  // am1:a0:a1:a2 += chi:clo placed with its bit 61 at stream position B; returns the carry out of
  // am1 (which needs am1 = 2^32 - 1, so almost never happens)
  __device__ __forceinline__ uint32_t add(uint32_t clo, uint32_t chi) {
    uint32_t cy;
    asm("{\n\t.reg .u32 x0, x1, x2;\n\t"
        "shf.l.wrap.b32 x2, 0, %5, %7;\n\t"
        "shf.l.wrap.b32 x1, %5, %6, %7;\n\t"
        "shf.l.wrap.b32 x0, %6, 0, %7;\n\t"
        "add.cc.u32 %2, %2, x2;\n\t"
        "addc.cc.u32 %1, %1, x1;\n\t"
        "addc.cc.u32 %0, %0, x0;\n\t"
        "addc.cc.u32 %4, %4, 0;\n\t"
        "addc.u32 %3, 0, 0;\n\t}"
        : "+r"(a0), "+r"(a1), "+r"(a2), "=r"(cy), "+r"(am1)
        : "r"(clo), "r"(chi), "r"(sh));
    return cy;
  }
  // one token; a completed word goes to the ring
  template <bool CHECK>
  __device__ __forceinline__ void token(uint32_t s, uint32_t f, int P) {
    if (CHECK) {
      const uint32_t u = f - 1u;
      chk |= s | u | (s + u);
    }
    uint32_t clo, chi, plo, phi;
    asm("{\n\t.reg .u64 c;\n\tmul.wide.u32 c, %2, %3;\n\tmov.b64 {%0, %1}, c;\n\tmad.lo.u32 %1, %4, %3, %1;\n\t}"
        : "=r"(clo), "=r"(chi)
        : "r"(rlo), "r"(s), "r"(rhi));
    if (add(clo, chi)) carry();
    asm("{\n\t.reg .u64 c;\n\tmul.wide.u32 c, %2, %3;\n\tmov.b64 {%0, %1}, c;\n\tmad.lo.u32 %1, %4, %3, %1;\n\t}"
        : "=r"(plo), "=r"(phi)
        : "r"(rlo), "r"(f), "r"(rhi));
    // k = 62 - bitlen(r f): clz of the high word less 2, plus 1 for r f = 2^62 (f = T). For any
    // input k lies in [0, 30], so sh and w stay bounded whatever the pairs hold. Unchecked pairs
    // (the encode path's, from the CDF kernels) have f < T, so r f < 2^62 and the correction is
    // never needed there; garbage pairs then give k in [-2, 30], with sh and w still bounded.
    // (k + 2 is kept, so that P - k and sh - k are each one add of a constant)
    int32_t z;
    asm("clz.b32 %0, %1;" : "=r"(z) : "r"(phi));
    if (CHECK) z += (int32_t)(phi >> 30);
    const int32_t s2 = (P + 2) - z;  // P - k, in [0, P] for valid pairs
    asm("shf.r.wrap.b32 %0, %1, %2, %3;" : "=r"(rlo) : "r"(plo), "r"(phi), "r"(s2));
    asm("shr.u32 %0, %1, %2;" : "=r"(rhi) : "r"(phi), "r"(s2));
    sh = (sh + 2) - z;
    const bool full = sh < 0;
    // the completed word before a0 leaves for the ring (words -2 and -1, which the first two
    // completions retire, land in ring slots that are rewritten before any read; they are
    // nonzero only after a carry past word 0, impossible for valid pairs, so only the checked
    // form looks at them)
    if (full) {
      ring_st(w - 1, am1);
      if (CHECK) nz |= w <= 0 ? am1 : 0u;
    }
    am1 = full ? a0 : am1;
    a0 = full ? a1 : a0;
    a1 = full ? a2 : a1;
    a2 = full ? 0u : a2;
    sh += full ? 32 : 0;
    w += full ? 1 : 0;
  }
  // the completed 16-byte chunks of the ring to the slot, keeping at least the last completed
  // word in the ring: a carry out of a0 (not rare while the window's offset is small) then
  // lands in shared memory instead of a global read-modify-write of the slot. k <= 30 per token,
  // so at most 8 words complete per 8 tokens; two chunks leave at most 4 words behind, and at
  // most 12 of the ring's 16 are ever pending.
  template <int CHUNKS>
  __device__ __forceinline__ void flush() {
#pragma unroll
    for (int q = 0; q < CHUNKS; q++) {
      if (w - fw >= 5) {
        uint4 v;
        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "r"(ring + 4u * (uint32_t)(fw & (kRingWords - 1)))
                     : "memory");
        if ((uint32_t)(fw + 3) < max_words) *reinterpret_cast<uint4*>(word(fw)) = v;
        fw += 4;
      }
    }
  }
  // termination: v = ceil(L / 2^60) * 2^60, i.e. add 2^60 - 1 at B and keep the top B + 2 bits;
  // returns B + 2 and writes every remaining word
  __device__ __forceinline__ uint64_t finish() {
    if (add(0xFFFFFFFFu, 0x0FFFFFFFu)) carry();
    // am1 back into the ring (word w - 1), or, below word 0, checked to be zero like the words
    // below word 0 that completed earlier
    if (w >= 1) ring_st(w - 1, am1);
    else nz |= am1;
    overflow |= nz != 0u;
    const int32_t off = 34 - sh;
    int32_t nrem;  // bits of the code in a0 (and a1)
    uint64_t nbits;
    if (w < 0) {  // B < 3: a0 holds stream bits [-32, 0), zero for valid input
      overflow |= a0 != 0u;
      a0 = a1;
      a1 = a2;
      w = 0;
      nrem = off - 30;
      nbits = (uint64_t)nrem;
    } else {
      nrem = off + 2;
      nbits = (uint64_t)w * 32u + (uint64_t)nrem;
    }
    for (int32_t i = fw; i < w; i++)
      if ((uint32_t)i < max_words) *word(i) = ring_ld(i);
    if ((uint32_t)w < max_words) *word(w) = nrem >= 32 ? a0 : a0 & ~(0xFFFFFFFFu >> nrem);
    if (nrem > 32 && (uint32_t)(w + 1) < max_words) *word(w + 1) = a1 & ~(0xFFFFFFFFu >> (nrem - 32));
    // a valid code fits its slot; pairs that were not checked may yield any length, which must
    // not send the packing step past the slot
    const uint64_t cap_bits = (uint64_t)max_words * 32u;
    return nbits < cap_bits ? nbits : cap_bits;
  }
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// One stream per thread, pairs at start[w*stride_win + i*stride_pos] (lmgc_range_encode's general
// layout), loaded 8 tokens ahead. PT: P at compile time (0: P_rt). CHECK: validate the pairs (a
// window stops after the group holding an invalid pair, and the error word reports it).
template <int PT, bool CHECK>
__global__ void __launch_bounds__(kCoderThreads) k_range_encode(
    const uint32_t* __restrict__ start, const uint32_t* __restrict__ freq, int P_rt, int64_t n_win,
    int64_t win_tokens, const uint32_t* __restrict__ win_len, int64_t stride_win, int64_t stride_pos,
    uint8_t* __restrict__ slots, size_t slot_sz, uint32_t* __restrict__ bitlen, uint32_t* err) {
  __shared__ __align__(16) uint32_t rings[kCoderThreads * kRingStride];
  const int P = PT ? PT : P_rt;
  const uint32_t T = 1u << P;
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= n_win) return;
  int64_t n = win_len ? (int64_t)win_len[w] : win_tokens;
  bool bad = n > win_tokens;
  if (bad) n = 0;  // a window longer than its slot is not coded
  Stream<false> c;
  c.init(P, reinterpret_cast<uint32_t*>(slots + (size_t)w * slot_sz), (uint32_t)(slot_sz / 4),
         rings + threadIdx.x * kRingStride);
  constexpr int kPre = 8;
  const uint32_t* qs = start + w * stride_win;
  const uint32_t* qf = freq + w * stride_win;
  uint32_t bs[kPre], bf[kPre];
#pragma unroll
  for (int j = 0; j < kPre; j++) {
    bs[j] = j < n ? __ldcs(qs) : 0u;
    bf[j] = j < n ? __ldcs(qf) : 1u;
    qs += stride_pos;
    qf += stride_pos;
  }
  for (int64_t i0 = 0; i0 < n; i0 += kPre) {
    uint32_t cs[kPre], cf[kPre];
    const bool full_next = i0 + 2 * kPre <= n;
#pragma unroll
    for (int j = 0; j < kPre; j++) {
      cs[j] = bs[j];
      cf[j] = bf[j];
      if (full_next || i0 + kPre + j < n) {
        bs[j] = __ldcs(qs);
        bf[j] = __ldcs(qf);
      }
      qs += stride_pos;
      qf += stride_pos;
    }
    if (i0 + kPre <= n) {
#pragma unroll
      for (int j = 0; j < kPre; j++) c.template token<CHECK>(cs[j], cf[j], P);
    } else {
      const int jn = (int)(n - i0);
#pragma unroll
      for (int j = 0; j < kPre; j++)
        if (j < jn) c.template token<CHECK>(cs[j], cf[j], P);
    }
    c.template flush<2>();
    if (CHECK && c.chk >= T) break;
  }
  bitlen[w] = (uint32_t)c.finish();
  if (bad || c.overflow || (CHECK && c.chk >= T)) atomicOr(err, kErrCorrupt);
}

// Pairs in window tiles (the encode path): a warp codes the 32 windows of one tile column, whose
// 8-position groups are contiguous 1 KiB tiles of starts and of freqs. The warp stages them
// through a two-stage ring in shared memory with asynchronous 16-byte copies (every lane copies
// its share of each tile, so that a copy instruction of the warp covers 512 contiguous bytes):
// the copies of group g + 2 are issued once every lane has read group g's stage, and so have two
// groups of coding to land. (Kilobyte bulk copies completing on an mbarrier, one lane issuing,
// were 1-2% slower.) No register holds pairs ahead beyond the group being coded. The codes go to
// the block's interleaved slot table (the slots array holds whole 32-window tables).
template <int PT, bool CHECK>
__global__ void __launch_bounds__(kCoderThreads) k_range_encode_tiles(
    const uint32_t* __restrict__ start, const uint32_t* __restrict__ freq, int P_rt, int64_t n_win,
    int64_t win_tokens, const uint32_t* __restrict__ win_len, uint8_t* __restrict__ slots, size_t slot_sz,
    uint32_t* __restrict__ bitlen, uint32_t* err) {
  constexpr int kWarps = kCoderThreads / 32;
  __shared__ __align__(16) uint32_t rings[kCoderThreads * kRingStride];
  __shared__ __align__(128) uint32_t tiles[kWarps][2][2][256];  // [warp][stage][start, freq][32 x 8]
  const int P = PT ? PT : P_rt;
  const uint32_t T = 1u << P;
  const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5;
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t w0 = w - lane;  // the tile column's first window
  if (w0 >= n_win) return;      // warp-uniform
  const bool live = w < n_win;
  int64_t n = live ? (win_len ? (int64_t)win_len[w] : win_tokens) : 0;
  const bool bad = n > win_tokens;
  if (bad) n = 0;  // a window longer than its slot is not coded
  const int64_t groups = pair_tile_groups(win_tokens);
  int64_t g_all = (n + 7) >> 3;  // groups any window of the warp codes (warp-uniform after the max)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) g_all = max(g_all, (int64_t)__shfl_xor_sync(0xffffffffu, (long long)g_all, o));
  Stream<true> c;
  c.init(P, reinterpret_cast<uint32_t*>(slots + (size_t)w0 * slot_sz), (uint32_t)(slot_sz / 4),
         rings + threadIdx.x * kRingStride, (uint32_t)lane);
  const int64_t col = pair_tile_index(w0, 0, groups);  // element of the column's first tile
  const uint32_t* ts = start + col;
  const uint32_t* tf = freq + col;
  // Each lane copies 16 bytes of each half kilobyte of a group's two tiles (every copy
  // instruction of the warp covers 512 contiguous bytes); a lane's own 32 bytes of an array thus
  // come from two other lanes, and __syncwarp after the wait makes them visible.
  const uint32_t stage0 = smem_addr(tiles[wp][0][0]);  // stage t, array a at + (2 t + a) KiB
  auto issue = [&](int64_t gg) {
    if (gg < g_all) {
      const uint32_t d = stage0 + (uint32_t)(gg & 1) * 2048u + 16u * (uint32_t)lane;
      const uint32_t* src_s = ts + (gg << 8) + 4 * lane;
      const uint32_t* src_f = tf + (gg << 8) + 4 * lane;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src_s) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d + 512u), "l"(src_s + 128) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d + 1024u), "l"(src_f) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d + 1536u), "l"(src_f + 128) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  issue(0);
  issue(1);
  const bool ok = true;
  bool stopped = false;
  for (int64_t g = 0; g < g_all; g++) {
    const int st = (int)(g & 1);
    asm volatile("cp.async.wait_group 1;" ::: "memory");  // this lane's copies of group g
    __syncwarp();                                          // and every other lane's
    const uint4* qs = reinterpret_cast<const uint4*>(tiles[wp][st][0] + 8 * lane);
    const uint4* qf = reinterpret_cast<const uint4*>(tiles[wp][st][1] + 8 * lane);
    const uint4 s0 = qs[0], s1 = qs[1], f0 = qf[0], f1 = qf[1];
    const uint32_t cs[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
    const uint32_t cf[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
    __syncwarp();  // every lane has read the stage
    issue(g + 2);
    if (!stopped && 8 * g < n) {
      if (8 * g + 8 <= n) {
#pragma unroll
        for (int j = 0; j < 8; j++) c.template token<CHECK>(cs[j], cf[j], P);
      } else {
        const int jn = (int)(n - 8 * g);
#pragma unroll
        for (int j = 0; j < 8; j++)
          if (j < jn) c.template token<CHECK>(cs[j], cf[j], P);
      }
      c.template flush<2>();
      if (CHECK && c.chk >= T) stopped = true;
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  if (!live) return;
  bitlen[w] = (uint32_t)c.finish();
  if (bad || !ok || c.overflow || (CHECK && c.chk >= T)) atomicOr(err, kErrCorrupt);
}

template <bool CHECK>
static void launch_coder(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                         const uint32_t* win_len, int64_t stride_win, int64_t stride_pos, uint8_t* slots,
                         size_t slot_sz, uint32_t* bitlen, uint32_t* err, cudaStream_t s) {
  const unsigned g = (unsigned)((n_win + kCoderThreads - 1) / kCoderThreads);
  if (P == 24)
    k_range_encode<24, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, stride_win,
                                                          stride_pos, slots, slot_sz, bitlen, err);
  else if (P == 16)
    k_range_encode<16, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, stride_win,
                                                          stride_pos, slots, slot_sz, bitlen, err);
  else
    k_range_encode<0, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, stride_win,
                                                         stride_pos, slots, slot_sz, bitlen, err);
}

template <bool CHECK>
static void launch_coder_tiles(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                               const uint32_t* win_len, uint8_t* slots, size_t slot_sz, uint32_t* bitlen,
                               uint32_t* err, cudaStream_t s) {
  const unsigned g = (unsigned)((n_win + kCoderThreads - 1) / kCoderThreads);
  if (P == 24)
    k_range_encode_tiles<24, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, slots,
                                                                slot_sz, bitlen, err);
  else if (P == 16)
    k_range_encode_tiles<16, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, slots,
                                                                slot_sz, bitlen, err);
  else
    k_range_encode_tiles<0, CHECK><<<g, kCoderThreads, 0, s>>>(start, freq, P, n_win, win_tokens, win_len, slots,
                                                               slot_sz, bitlen, err);
}

void launch_range_encode(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                         const uint32_t* win_len, int64_t stride_win, int64_t stride_pos, uint8_t* slots,
                         size_t slot_sz, uint32_t* bitlen, uint32_t* err, cudaStream_t s, bool tiled, bool check) {
  if (n_win <= 0) return;
  note_launch();
  if (tiled) {
    if (check) launch_coder_tiles<true>(start, freq, P, n_win, win_tokens, win_len, slots, slot_sz, bitlen, err, s);
    else launch_coder_tiles<false>(start, freq, P, n_win, win_tokens, win_len, slots, slot_sz, bitlen, err, s);
  } else {
    launch_coder<true>(start, freq, P, n_win, win_tokens, win_len, stride_win, stride_pos, slots, slot_sz, bitlen,
                       err, s);
  }
}

// ------------------------------------------------------------------------------------------
// Container payload: exclusive scan of the code byte lengths (one block), then each window's
// ceil(bitlen/8) bytes copied from its slot (words in native order) to its offset.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_scan_lengths(const uint32_t* __restrict__ bitlen, int64_t n,
                                                       uint64_t* __restrict__ off) {
  __shared__ uint64_t wsum[32];
  __shared__ uint64_t carry;
  const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
  if (t == 0) carry = 0;
  __syncthreads();
  for (int64_t base = 0; base < n; base += 1024) {
    int64_t i = base + t;
    uint64_t v = i < n ? (uint64_t)((bitlen[i] + 7u) / 8u) : 0ull;
    uint64_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint64_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[wid] = x;
    __syncthreads();
    if (wid == 0) {
      uint64_t y = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        uint64_t z = __shfl_up_sync(0xffffffffu, y, o);
        if (lane >= o) y += z;
      }
      wsum[lane] = y;
    }
    __syncthreads();
    uint64_t excl = carry + (wid > 0 ? wsum[wid - 1] : 0ull) + x - v;
    if (i < n) off[i] = excl;
    __syncthreads();
    if (t == 1023) carry = excl + v;
    __syncthreads();
  }
  if (t == 0) off[n] = carry;
}

__global__ void k_copy_codes(const uint8_t* __restrict__ slots, size_t slot_sz, const uint32_t* __restrict__ bitlen,
                             const uint64_t* __restrict__ off, int64_t n, uint8_t* __restrict__ out, bool ilv) {
  for (int64_t w = blockIdx.x; w < n; w += gridDim.x) {
    const uint32_t nb = (bitlen[w] + 7u) / 8u;
    uint8_t* dst = out + off[w];
    // slot words are in native (little-endian) byte order; the code's bytes go most significant first
    if (!ilv) {
      const uint8_t* src = slots + (size_t)w * slot_sz;
      for (uint32_t b = threadIdx.x; b < nb; b += blockDim.x) dst[b] = src[b ^ 3u];
    } else {
      // the warp's table: 16-byte chunk c of window w at ((c * 32 + w % 32) * 16) from its base
      const uint8_t* base = slots + (size_t)(w & ~(int64_t)31) * slot_sz;
      const uint32_t col = (uint32_t)(w & 31);
      for (uint32_t b = threadIdx.x; b < nb; b += blockDim.x)
        dst[b] = base[((size_t)(b >> 4) * 32u + col) * 16u + ((b & 15u) ^ 3u)];
    }
  }
}

void launch_pack_codes(const uint8_t* slots, size_t slot_sz, const uint32_t* bitlen, int64_t n_win, uint64_t* offsets,
                       uint8_t* out, cudaStream_t s, bool interleaved) {
  if (n_win <= 0) return;
  note_launch();
  k_scan_lengths<<<1, 1024, 0, s>>>(bitlen, n_win, offsets);
  if (out) {
    unsigned blocks = (unsigned)std::min<int64_t>(n_win, 152 * 16);
    note_launch();
    k_copy_codes<<<blocks, 128, 0, s>>>(slots, slot_sz, bitlen, offsets, n_win, out, interleaved);
  }
}

// ------------------------------------------------------------------------------------------
// Token checksums of the container: CRC-32 (IEEE 802.3, reflected polynomial 0xEDB88320, initial
// value and final xor 0xFFFFFFFF) of each window's token ids as little-endian u16 bytes. One
// thread per window, one table lookup per byte; the 256-entry table is built in shared memory
// from the polynomial by every block.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t crc_byte(const uint32_t* tab, uint32_t c, uint32_t b) {
  return tab[(c ^ b) & 0xFFu] ^ (c >> 8);
}

__global__ void __launch_bounds__(256) k_window_crc(const uint16_t* __restrict__ tok, int64_t stride,
                                                    const uint32_t* __restrict__ len, int64_t n_win,
                                                    uint32_t* __restrict__ out) {
  __shared__ uint32_t tab[256];
  {
    uint32_t c = threadIdx.x;
    for (int k = 0; k < 8; k++) c = (c & 1u) ? 0xEDB88320u ^ (c >> 1) : c >> 1;
    tab[threadIdx.x] = c;
  }
  __syncthreads();
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= n_win) return;
  const uint16_t* t = tok + w * stride;
  const uint32_t n = len[w];
  uint32_t c = 0xFFFFFFFFu, i = 0;
  if ((reinterpret_cast<uintptr_t>(t) & 15) == 0) {
    for (; i + 8 <= n; i += 8) {
      const uint4 v = *reinterpret_cast<const uint4*>(t + i);
      const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int k = 0; k < 4; k++)
#pragma unroll
        for (int b = 0; b < 4; b++) c = crc_byte(tab, c, (words[k] >> (8 * b)) & 0xFFu);
    }
  }
  for (; i < n; i++) {
    c = crc_byte(tab, c, t[i] & 0xFFu);
    c = crc_byte(tab, c, t[i] >> 8);
  }
  out[w] = c ^ 0xFFFFFFFFu;
}

void launch_window_crc(const uint16_t* tok, int64_t stride, const uint32_t* len, int64_t n_win, uint32_t* out,
                       cudaStream_t s) {
  if (n_win <= 0) return;
  note_launch();
  k_window_crc<<<(unsigned)((n_win + 255) / 256), 256, 0, s>>>(tok, stride, len, n_win, out);
}

// ------------------------------------------------------------------------------------------
// Allocation-free variant of lmgc_range_encode.
//
// Some callers cannot allocate device memory at all: a process whose device memory is held
// entirely by another allocator, or a latency-critical path on which cudaMalloc / cudaFree
// (which may synchronise the device) are not allowed. For them the coder's scratch -- one code
// slot per window, the payload offsets and an error word -- lives in the fixed array below
// instead of being allocated per call. Every GPU that loads this library keeps the array
// (kNoAllocScratchBytes) until the process exits.
// ------------------------------------------------------------------------------------------
constexpr size_t kNoAllocScratchBytes = 64ull << 20;  // 64 MiB
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
uint8_t* g_noalloc_ptr[kMaxDevices] = {};  // device address of the array, per device

// In host code g_noalloc_scratch names a host-side stand-in, not device memory: the device
// address is looked up once per device, with that device current.
lmgc_status noalloc_scratch(uint8_t** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(nullptr, LMGC_ERR_INVALID, "lmgc_range_encode_noalloc: device id");
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: cudaGetSymbolAddress");
    g_noalloc_ptr[dev] = (uint8_t*)p;
  }
  *out = g_noalloc_ptr[dev];
  return LMGC_OK;
}
}  // namespace

}  // namespace lmgc

extern "C" lmgc_status lmgc_range_encode_noalloc(const uint32_t* d_start, const uint32_t* d_freq, int cdf_bits,
                                                 size_t n_win, size_t win_tokens, const uint32_t* d_win_len,
                                                 size_t stride_win, size_t stride_pos, uint8_t* d_out, size_t cap,
                                                 size_t* out_bytes, uint32_t* d_bitlen, lmgc_stream stream) {
  using namespace lmgc;
  if (!out_bytes || (n_win && (!d_start || !d_freq || !d_bitlen)))
    return fail(nullptr, LMGC_ERR_INVALID, "lmgc_range_encode_noalloc: null argument");
  if (cdf_bits < 1 || cdf_bits > 30)
    return fail(nullptr, LMGC_ERR_INVALID, "lmgc_range_encode_noalloc: cdf_bits must be in 1..30");
  *out_bytes = 0;
  if (n_win == 0) return LMGC_OK;
  // a window longer than this cannot fit in the array whatever n_win is; bounding it first also
  // keeps slot_bytes' size arithmetic from wrapping
  if (win_tokens > (kNoAllocScratchBytes * 8) / (size_t)cdf_bits)
    return fail(nullptr, LMGC_ERR_INVALID,
                "lmgc_range_encode_noalloc: win_tokens * cdf_bits exceeds the fixed maximum of " +
                    std::to_string(kNoAllocScratchBytes) + " bytes of scratch");
  // scratch layout: [0, 256) error word | offsets [n_win + 1] u64 | one code slot per window
  const size_t slot = slot_bytes(win_tokens, cdf_bits);
  const size_t off_bytes = ((n_win + 1) * 8 + 255) / 256 * 256;
  const double need = 256.0 + (double)off_bytes + (double)slot * (double)n_win;
  if (need > (double)kNoAllocScratchBytes)
    return fail(nullptr, LMGC_ERR_INVALID,
                "lmgc_range_encode_noalloc: needs " + std::to_string((unsigned long long)need) +
                    " bytes of scratch (n_win * slot + offsets); the fixed maximum is " +
                    std::to_string(kNoAllocScratchBytes) + " bytes");
  uint8_t* base = nullptr;
  lmgc_status st = noalloc_scratch(&base);
  if (st != LMGC_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  uint32_t* derr = (uint32_t*)base;
  uint64_t* offs = (uint64_t*)(base + 256);
  uint8_t* slots = base + 256 + off_bytes;
  // the array keeps the previous call's contents: only the error word must start at zero (the
  // slots are written before they are read and the offsets are recomputed)
  cudaError_t e = cudaMemsetAsync(derr, 0, 4, s);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: clear");
  launch_range_encode(d_start, d_freq, cdf_bits, (int64_t)n_win, (int64_t)win_tokens, d_win_len,
                      (int64_t)stride_win, (int64_t)stride_pos, slots, slot, d_bitlen, derr, s);
  launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, nullptr, s, false);
  // a failed launch must not let the previous call's total (still in the array) be read back
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: launch");
  uint64_t total = 0;
  uint32_t herr = 0;
  e = cudaMemcpyAsync(&total, offs + n_win, 8, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, derr, 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc");
  if (herr) return fail(nullptr, LMGC_ERR_INVALID, "lmgc_range_encode_noalloc: invalid (start, freq) or window length");
  *out_bytes = total;
  if (cap < total) return fail(nullptr, LMGC_ERR_NO_SPACE, "lmgc_range_encode_noalloc: output too small");
  launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, d_out, s, false);
  e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: pack");
  return LMGC_OK;
}
