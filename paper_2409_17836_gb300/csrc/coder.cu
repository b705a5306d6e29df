// coder.cu -- the arithmetic coder (Sec. 2 "Arithmetic coding") in exact integer form, one
// independent stream per window (Sec. 3 "Compression": each window is coded from its own BOS).
//
// Per stream: R = 2^62, L = 0, B = 0; per token (s = start, f = freq, T = 2^P):
//   r = R >> P;  L += r*s;  R = r*f;  k = max(0, 62 - bitlen(R));  R <<= k;  L <<= k;  B += k
// and the code is the top B + 2 bits of v = ceil(L / 2^60) * 2^60 (v lies in [L, L + R) because
// R >= 2^61), most significant bit first.
//
// The range R depends only on the freq sequence; L is the only unbounded quantity. A thread keeps
// the low 62 bits of L in a register; the bits shifted above them are emitted into a 64-bit
// accumulator and leave in 32-bit words to the stream's own scratch slot. A carry out of the
// low 62 bits increments the emitted bits: in the accumulator, or -- when the accumulator was all
// ones -- in the already written words of this stream's slot (never beyond word 0: L + R stays
// below 2^(B+62)). The carry walk is bounded by the slot length.
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

struct Emitter {
  uint32_t* slot;   // stream words (stored big-endian so the bytes are in stream order)
  uint32_t wpos;    // words written
  uint32_t max_words;
  uint64_t acc;     // pending emitted bits, right-aligned
  int nacc;         // number of pending bits (< 32 after each flush)
  bool overflow;

  __device__ __forceinline__ void carry() {
    acc += 1;
    if ((acc >> nacc) != 0) {  // pending bits were all ones: carry into written words
      acc = 0;
      int64_t i = (int64_t)wpos - 1;
      for (; i >= 0; --i) {
        uint32_t v = bswap32(slot[i]) + 1u;
        slot[i] = bswap32(v);
        if (v != 0u) break;
      }
      if (i < 0) overflow = true;  // impossible for valid input; reported, not propagated
    }
  }
  __device__ __forceinline__ void put(uint64_t bits, int k) {  // append k (<= 32) bits
    acc = (acc << k) | bits;
    nacc += k;
    if (nacc >= 32) {
      uint32_t w = (uint32_t)(acc >> (nacc - 32));
      if (wpos < max_words) slot[wpos] = bswap32(w);
      else overflow = true;
      wpos++;
      nacc -= 32;
      acc &= (nacc > 0) ? ((1ull << nacc) - 1ull) : 0ull;
    }
  }
};

__global__ void __launch_bounds__(128) k_range_encode(const uint32_t* __restrict__ start,
                                                      const uint32_t* __restrict__ freq, int P, int64_t n_win,
                                                      int64_t win_tokens, const uint32_t* __restrict__ win_len,
                                                      int64_t stride_win, int64_t stride_pos, uint8_t* __restrict__ slots,
                                                      size_t slot_sz, uint32_t* __restrict__ bitlen, uint32_t* err) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= n_win) return;
  const int64_t n = win_len ? (int64_t)win_len[w] : win_tokens;
  const uint64_t mask62 = (1ull << 62) - 1ull;
  const uint64_t T = 1ull << P;
  Emitter em;
  em.slot = reinterpret_cast<uint32_t*>(slots + (size_t)w * slot_sz);
  em.wpos = 0;
  em.max_words = (uint32_t)(slot_sz / 4);
  em.acc = 0;
  em.nacc = 0;
  em.overflow = false;
  uint64_t R = 1ull << 62, L = 0, B = 0;
  bool bad = n > win_tokens;
  const uint32_t* ps = start + w * stride_win;
  const uint32_t* pf = freq + w * stride_win;
  // the pairs of the next kPre tokens are loaded ahead so their latency overlaps the serial chain
  constexpr int kPre = 8;
  uint32_t bs[kPre], bf[kPre];
#pragma unroll
  for (int j = 0; j < kPre; j++) {
    bs[j] = j < n ? __ldcs(ps + j * stride_pos) : 0u;
    bf[j] = j < n ? __ldcs(pf + j * stride_pos) : 1u;
  }
  for (int64_t i0 = 0; i0 < n && !bad; i0 += kPre) {
    uint32_t cs[kPre], cf[kPre];
#pragma unroll
    for (int j = 0; j < kPre; j++) {
      cs[j] = bs[j];
      cf[j] = bf[j];
      const int64_t nx = i0 + kPre + j;
      bs[j] = nx < n ? __ldcs(ps + nx * stride_pos) : 0u;
      bf[j] = nx < n ? __ldcs(pf + nx * stride_pos) : 1u;
    }
#pragma unroll
  for (int j = 0; j < kPre; j++) {
    if (i0 + j >= n) break;
    const uint64_t s = cs[j];
    const uint64_t f = cf[j];
    if (f == 0 || s + f > T) {
      bad = true;
      break;
    }
    const uint64_t r = R >> P;
    L += r * s;  // < 2^63
    if (L >> 62) {
      L &= mask62;
      em.carry();
    }
    R = r * f;
    const int k = __clzll((long long)R) - 2;  // 62 - bitlen(R) >= 0 since R < 2^62
    if (k > 0) {
      em.put(L >> (62 - k), k);
      L = (L << k) & mask62;
      R <<= k;
      B += (uint64_t)k;
    }
  }
  }
  // termination: v = ceil(L / 2^60) * 2^60; emit its top 2 bits of the low 62
  L += (1ull << 60) - 1ull;
  if (L >> 62) {
    L &= mask62;
    em.carry();
  }
  em.put(L >> 60, 2);
  if (em.nacc > 0) {
    uint32_t wv = (uint32_t)(em.acc << (32 - em.nacc));
    if (em.wpos < em.max_words) em.slot[em.wpos] = bswap32(wv);
    else em.overflow = true;
  }
  bitlen[w] = (uint32_t)(B + 2);
  if (bad || em.overflow) atomicOr(err, kErrCorrupt);
}

void launch_range_encode(const uint32_t* start, const uint32_t* freq, int P, int64_t n_win, int64_t win_tokens,
                         const uint32_t* win_len, int64_t stride_win, int64_t stride_pos, uint8_t* slots,
                         size_t slot_sz, uint32_t* bitlen, uint32_t* err, cudaStream_t s) {
  if (n_win <= 0) return;
  note_launch();
  k_range_encode<<<(unsigned)((n_win + 127) / 128), 128, 0, s>>>(start, freq, P, n_win, win_tokens, win_len,
                                                                  stride_win, stride_pos, slots, slot_sz, bitlen, err);
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
  uint64_t total = 0;
  uint32_t herr = 0;
  cudaMemcpyAsync(&total, offs + n_win, 8, cudaMemcpyDeviceToHost, s);
  cudaMemcpyAsync(&herr, derr, 4, cudaMemcpyDeviceToHost, s);
  e = cudaStreamSynchronize(s);
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
