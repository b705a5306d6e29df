// coder.cu -- the arithmetic coder (Sec. 3 "Arithmetic coding") in exact integer form, one
// independent stream per window (Sec. 4 "Compression": each window is coded from its own BOS).
//
// Per stream: R = 2^62, L = 0, B = 0; per token (s = start, f = freq, T = 2^P):
//   r = R >> P;  L += r*s;  R = r*f;  k = max(0, 62 - bitlen(R));  R <<= k;  L <<= k;  B += k
// and the code is the top B + 2 bits of v = ceil(L / 2^60) * 2^60 (v lies in [L, L + R) because
// R >= 2^61), most significant bit first.
//
// The range R depends only on the freq sequence; L is the only unbounded quantity. A thread keeps
// the low 62 bits of L in a register (as 4 L, so that the carry out of them is the carry out of
// a 64-bit add); the bits shifted above them collect in a 32-bit pending word and leave in 32-bit
// words to the stream's own scratch slot. A carry out of the low 62 bits increments the emitted
// bits: the pending ones, or -- when they were all ones -- the already written words of this
// stream's slot (never beyond word 0: L + R stays below 2^(B+62)). The carry walk is bounded by
// the slot length. All shifts are 32-bit funnel shifts by less than 32 (k <= P <= 30 per token).
//
// Layout: one stream per thread, 32 windows per warp. Pairs are read at
// start[w*stride_win + i*stride_pos]; with the encode path's position-major layout
// (stride_win = 1) a warp's 32 loads of token i are one 128-byte transaction.
#include <algorithm>
#include <mutex>
#include <string>

#include "lmgc_internal.cuh"

namespace lmgc {

size_t slot_bytes(size_t win_tokens, int P) {
  size_t bits = win_tokens * (size_t)P + 2;
  size_t words = (bits + 31) / 32 + 1;
  return ((words * 4 + 15) / 16) * 16;
}

__device__ __forceinline__ uint32_t bswap32(uint32_t x) { return __byte_perm(x, 0, 0x0123); }

// 64-bit add with the carry out of bit 63
__device__ __forceinline__ uint64_t add_carry(uint64_t a, uint64_t b, uint32_t& c) {
  uint32_t lo, hi;
  asm("add.cc.u32 %0, %3, %5;\n\taddc.cc.u32 %1, %4, %6;\n\taddc.u32 %2, 0, 0;"
      : "=r"(lo), "=r"(hi), "=r"(c)
      : "r"((uint32_t)a), "r"((uint32_t)(a >> 32)), "r"((uint32_t)b), "r"((uint32_t)(b >> 32)));
  return ((uint64_t)hi << 32) | lo;
}

// One stream's coder state in 32-bit pieces. L is held as L4 = 4 L (its 62 bits at the top of a
// 64-bit word, so a carry out of bit 62 of L is the carry out of the 64-bit add); the emitted bits
// not yet written form `acc` (nacc < 32 bits, right-aligned). Every shift is a 32-bit (funnel)
// shift by less than 32: k <= P <= 30 bits move per token.
struct Coder {
  uint32_t R_hi, R_lo;
  uint64_t L4;
  uint32_t acc, nacc, wpos, max_words;
  uint32_t* slot;  // stream words, big-endian
  bool overflow;

  __device__ __forceinline__ void write(uint32_t wv) {
    if (wpos < max_words) slot[wpos] = bswap32(wv);
    else overflow = true;
    wpos++;
  }
  // +cy (0 or 1) into the emitted bits: the pending ones, else (all ones) the written words
  __device__ __forceinline__ void carry(uint32_t cy) {
    acc += cy;
    if ((acc >> nacc) != 0u) {  // only when cy = 1 and the pending bits were all ones
      acc = 0u;
      int64_t i = (int64_t)wpos - 1;
      for (; i >= 0; --i) {
        uint32_t v = bswap32(slot[i]) + 1u;
        slot[i] = bswap32(v);
        if (v != 0u) break;
      }
      if (i < 0) overflow = true;  // impossible for valid input; reported, not propagated
    }
  }
  // move the top k (< 32) bits of L4 to the pending bits; L4 and R shift left by k
  __device__ __forceinline__ void shift_out(uint32_t k) {
    const uint32_t l_hi = (uint32_t)(L4 >> 32), l_lo = (uint32_t)L4;
    const uint32_t a_hi = __funnelshift_l(acc, 0u, k);            // acc >> (32 - k), 0 for k = 0
    const uint32_t a_lo = (acc << k) | __funnelshift_l(l_hi, 0u, k);
    L4 = ((uint64_t)__funnelshift_l(l_lo, l_hi, k) << 32) | (l_lo << k);
    R_hi = __funnelshift_l(R_lo, R_hi, k);
    R_lo <<= k;
    // a full word leaves when 32 or more bits are pending (a_hi = 0 otherwise); no branch
    const bool full = nacc + k >= 32u;
    nacc = full ? nacc + k - 32u : nacc + k;
    const uint32_t wv = __funnelshift_r(a_lo, a_hi, nacc);  // the top 32 of the nacc + 32 pending bits
    const bool in_slot = wpos < max_words;
    if (full && in_slot) slot[wpos] = bswap32(wv);
    overflow |= full && !in_slot;
    wpos += full ? 1u : 0u;
    acc = full ? (a_lo & ((1u << nacc) - 1u)) : a_lo;
  }
};

// Per token (s = start, f = freq, T = 2^P): r = R >> P; L4 += 4 r s (carry -> emitted bits);
// R = r f; k = max(0, clz(R) - 2); shift_out(k). R >= 2^(61 - P) after the multiply, so for
// P <= 29 its high word is nonzero (HI32: a 32-bit count of leading zeros).
template <bool HI32>
__device__ __forceinline__ void code_token(Coder& c, uint32_t s, uint32_t f, int P, uint32_t T, bool& bad) {
  // 0 < f <= T and s + f <= T; an invalid pair stops the stream after its group (the arithmetic
  // stays bounded meanwhile: writes are slot-checked and the carry walk stops at word 0)
  bad |= (f - 1u >= T) | (s > T - f);
  const uint32_t r_lo = __funnelshift_r(c.R_lo, c.R_hi, (uint32_t)P), r_hi = c.R_hi >> P;
  const uint64_t r = ((uint64_t)r_hi << 32) | r_lo;
  uint32_t cy;
  c.L4 = add_carry(c.L4, r * (uint64_t)(s << 2), cy);  // r s < 2^62, so 4 r s < 2^64
  c.carry(cy);
  const uint64_t Rn = r * (uint64_t)f;
  c.R_hi = (uint32_t)(Rn >> 32);
  c.R_lo = (uint32_t)Rn;
  int k = (HI32 ? __clz((int)c.R_hi) : __clzll((long long)Rn)) - 2;
  k = max(k, 0);                // R = 2^62 (f = T) needs no shift
  if (!HI32) k = min(k, 31);    // only an invalid f = 0 reaches past P
  c.shift_out((uint32_t)k);
}

template <bool HI32>
__global__ void __launch_bounds__(128) k_range_encode(const uint32_t* __restrict__ start,
                                                      const uint32_t* __restrict__ freq, int P, int64_t n_win,
                                                      int64_t win_tokens, const uint32_t* __restrict__ win_len,
                                                      int64_t stride_win, int64_t stride_pos, uint8_t* __restrict__ slots,
                                                      size_t slot_sz, uint32_t* __restrict__ bitlen, uint32_t* err) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= n_win) return;
  const int64_t n = win_len ? (int64_t)win_len[w] : win_tokens;
  const uint32_t T = 1u << P;
  Coder c;
  c.R_hi = 1u << 30;  // R = 2^62
  c.R_lo = 0u;
  c.L4 = 0ull;
  c.acc = 0u;
  c.nacc = 0u;
  c.wpos = 0u;
  c.max_words = (uint32_t)(slot_sz / 4);
  c.slot = reinterpret_cast<uint32_t*>(slots + (size_t)w * slot_sz);
  c.overflow = false;
  bool bad = n > win_tokens;
  // the pairs of the next kPre tokens are loaded ahead so their latency overlaps the serial chain;
  // the load pointers advance by the position stride
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
  for (int64_t i0 = 0; i0 < n && !bad; i0 += kPre) {
    uint32_t cs[kPre], cf[kPre];
    const bool full_next = i0 + 2 * kPre <= n;
#pragma unroll
    for (int j = 0; j < kPre; j++) {
      cs[j] = bs[j];
      cf[j] = bf[j];
      if (full_next || i0 + kPre + j < n) {
        bs[j] = __ldcs(qs);
        bf[j] = __ldcs(qf);
      } else {
        bs[j] = 0u;
        bf[j] = 1u;
      }
      qs += stride_pos;
      qf += stride_pos;
    }
    if (i0 + kPre <= n) {
#pragma unroll
      for (int j = 0; j < kPre; j++) code_token<HI32>(c, cs[j], cf[j], P, T, bad);
    } else {
      const int jn = (int)(n - i0);
#pragma unroll
      for (int j = 0; j < kPre; j++)
        if (j < jn) code_token<HI32>(c, cs[j], cf[j], P, T, bad);
    }
  }
  // termination: v = ceil(L / 2^60) * 2^60; emit its top 2 bits of the low 62
  {
    uint32_t cy;
    c.L4 = add_carry(c.L4, ((1ull << 60) - 1ull) << 2, cy);
    c.carry(cy);
  }
  c.shift_out(2u);
  // every emitted bit went through the pending bits: B + 2 bits in all
  const uint64_t nbits = (uint64_t)c.wpos * 32u + c.nacc;
  if (c.nacc > 0u) c.write(c.acc << (32u - c.nacc));
  bitlen[w] = (uint32_t)nbits;
  if (bad || c.overflow) atomicOr(err, kErrCorrupt);
}

void launch_range_encode(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                         const uint32_t* win_len, int64_t stride_win, int64_t stride_pos, uint8_t* slots,
                         size_t slot_sz, uint32_t* bitlen, uint32_t* err, cudaStream_t s) {
  if (n_win <= 0) return;
  note_launch();
  if (P <= 29)
    k_range_encode<true><<<(unsigned)((n_win + 127) / 128), 128, 0, s>>>(start, freq, P, n_win, win_tokens, win_len,
                                                                        stride_win, stride_pos, slots, slot_sz, bitlen,
                                                                        err);
  else
    k_range_encode<false><<<(unsigned)((n_win + 127) / 128), 128, 0, s>>>(start, freq, P, n_win, win_tokens, win_len,
                                                                         stride_win, stride_pos, slots, slot_sz, bitlen,
                                                                         err);
}

// ------------------------------------------------------------------------------------------
// Container payload: exclusive scan of the code byte lengths (one block), then each window's
// ceil(bitlen/8) bytes copied from its slot to its offset.
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
                             const uint64_t* __restrict__ off, int64_t n, uint8_t* __restrict__ out) {
  for (int64_t w = blockIdx.x; w < n; w += gridDim.x) {
    const uint32_t nb = (bitlen[w] + 7u) / 8u;
    const uint8_t* src = slots + (size_t)w * slot_sz;
    uint8_t* dst = out + off[w];
    for (uint32_t b = threadIdx.x; b < nb; b += blockDim.x) dst[b] = src[b];
  }
}

void launch_pack_codes(const uint8_t* slots, size_t slot_sz, const uint32_t* bitlen, int64_t n_win, uint64_t* offsets,
                       uint8_t* out, cudaStream_t s) {
  if (n_win <= 0) return;
  note_launch();
  k_scan_lengths<<<1, 1024, 0, s>>>(bitlen, n_win, offsets);
  if (out) {
    unsigned blocks = (unsigned)std::min<int64_t>(n_win, 152 * 16);
    note_launch();
    k_copy_codes<<<blocks, 128, 0, s>>>(slots, slot_sz, bitlen, offsets, n_win, out);
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
  launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, nullptr, s);
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
  launch_pack_codes(slots, slot, d_bitlen, (int64_t)n_win, offs, d_out, s);
  e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "lmgc_range_encode_noalloc: pack");
  return LMGC_OK;
}
