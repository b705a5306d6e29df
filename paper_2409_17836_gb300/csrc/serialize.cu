// serialize.cu -- fp32 / uint8 values -> hex-digit token ids with separators, and back.
//
// Sec. 4 "Serialization" and Fig. 1: each value's bits are cut into 4-bit groups, most
// significant first (for fp32: the sign and exponent nibbles lead), each group becomes one hex
// digit (token id = digit value 0..15), and a separator follows every value (' ' = 16,
// ',' = 17, ', ' = 17 16, ';' = 18, or none).
//
// HBM-bound: 4 B read + tpv * 2 B written per fp32 value. A block stages the tokens of 1024
// values in shared memory so that the writes leave as coalesced 16-byte vectors.
#include "lmgc_internal.cuh"

namespace lmgc {

int tokens_per_value(int input_kind, int sep_mode) {
  int nd = input_kind == LMGC_IN_F32 ? 8 : (input_kind == LMGC_IN_U8 ? 2 : -1);
  int ns = sep_mode == LMGC_SEP_NONE ? 0 : (sep_mode == LMGC_SEP_COMMA_SPACE ? 2 : 1);
  if (nd < 0 || sep_mode < 0 || sep_mode > 4) return -1;
  return nd + ns;
}

// Byte grouping (Sec. 5.3): bytes per value, and the group size (0 = one group per value).
static int64_t bytes_per_value(int input_kind) { return input_kind == LMGC_IN_F32 ? 4 : 1; }
static int sep_count(int sep_mode) { return sep_mode == LMGC_SEP_NONE ? 0 : (sep_mode == LMGC_SEP_COMMA_SPACE ? 2 : 1); }

int64_t serial_tokens(int input_kind, int sep_mode, int byte_group, int64_t n) {
  const int64_t bv = bytes_per_value(input_kind), g = byte_group ? byte_group : bv, nb = n * bv;
  return 2 * nb + sep_count(sep_mode) * ((nb + g - 1) / g);
}

int64_t serial_values(int input_kind, int sep_mode, int byte_group, int64_t n_tok) {
  // the layout repeats every lcm(bytes per value, group) bytes = pv values = pt tokens, and the
  // token count of q * pv + j values is q * pt + (the count of j values)
  const int64_t bv = bytes_per_value(input_kind), g = byte_group ? byte_group : bv;
  int64_t pb = bv;
  while (pb % g) pb += bv;
  const int64_t pv = pb / bv, pt = serial_tokens(input_kind, sep_mode, byte_group, pv);
  const int64_t q = n_tok / pt;
  for (int64_t j = 0; j < pv; j++)
    if (serial_tokens(input_kind, sep_mode, byte_group, q * pv + j) == n_tok) return q * pv + j;
  return -1;
}

bool serial_is_default(int input_kind, int byte_group, int byte_order) {
  return (byte_group == 0 || byte_group == bytes_per_value(input_kind)) && byte_order == 0;
}

static void sep_ids(int sep_mode, uint16_t* s0, uint16_t* s1) {
  switch (sep_mode) {
    case LMGC_SEP_SPACE: *s0 = kTokSpace; *s1 = 0; break;
    case LMGC_SEP_COMMA: *s0 = kTokComma; *s1 = 0; break;
    case LMGC_SEP_COMMA_SPACE: *s0 = kTokComma; *s1 = kTokSpace; break;
    case LMGC_SEP_SEMI: *s0 = kTokSemi; *s1 = 0; break;
    default: *s0 = 0; *s1 = 0; break;
  }
}

constexpr int kSerThreads = 256;
constexpr int kSerVals = 4 * kSerThreads;  // values per block

template <int ND, int NS, bool VEC>
__global__ void __launch_bounds__(kSerThreads) k_serialize(const void* __restrict__ in, int64_t n,
                                                           uint16_t* __restrict__ tok, uint16_t sep0,
                                                           uint16_t sep1) {
  constexpr int TPV = ND + NS;
  __shared__ __align__(16) uint16_t buf[kSerVals * TPV];
  const int t = threadIdx.x;
  const int64_t v0 = (int64_t)blockIdx.x * kSerVals;
  const int nv = (n - v0) < kSerVals ? (int)(n - v0) : kSerVals;
  uint32_t b[4];
  if (ND == 8) {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(in) + v0;
    if (VEC && nv == kSerVals) {
      uint4 q = __ldcs(reinterpret_cast<const uint4*>(src) + t);
      b[0] = q.x; b[1] = q.y; b[2] = q.z; b[3] = q.w;
    } else {
#pragma unroll
      for (int i = 0; i < 4; i++) b[i] = (4 * t + i < nv) ? src[4 * t + i] : 0u;
    }
  } else {
    const uint8_t* src = reinterpret_cast<const uint8_t*>(in) + v0;
    if (VEC && nv == kSerVals) {
      uint32_t q = __ldcs(reinterpret_cast<const unsigned int*>(src) + t);
#pragma unroll
      for (int i = 0; i < 4; i++) b[i] = (q >> (8 * i)) & 0xFFu;
    } else {
#pragma unroll
      for (int i = 0; i < 4; i++) b[i] = (4 * t + i < nv) ? src[4 * t + i] : 0u;
    }
  }
#pragma unroll
  for (int i = 0; i < 4; i++) {
    uint16_t* o = buf + (4 * t + i) * TPV;
#pragma unroll
    for (int j = 0; j < ND; j++) o[j] = (uint16_t)((b[i] >> (4 * (ND - 1 - j))) & 0xFu);
    if (NS >= 1) o[ND] = sep0;
    if (NS >= 2) o[ND + 1] = sep1;
  }
  __syncthreads();
  const int64_t tok0 = v0 * TPV;
  const int ntok = nv * TPV;
  uint16_t* dst = tok + tok0;
  if (VEC && nv == kSerVals) {
    // kSerVals * TPV * 2 bytes is a multiple of 16, and tok is 16-byte aligned (checked)
    const uint4* s4 = reinterpret_cast<const uint4*>(buf);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (int k = t; k < ntok / 8; k += kSerThreads) __stcs(d4 + k, s4[k]);
  } else {
    for (int k = t; k < ntok; k += kSerThreads) dst[k] = buf[k];
  }
}

template <int ND, int NS>
static void ser_dispatch(bool vec, const void* in, int64_t n, uint16_t* tok, uint16_t s0, uint16_t s1,
                         cudaStream_t s) {
  int64_t blocks = (n + kSerVals - 1) / kSerVals;
  if (vec) k_serialize<ND, NS, true><<<(unsigned)blocks, kSerThreads, 0, s>>>(in, n, tok, s0, s1);
  else k_serialize<ND, NS, false><<<(unsigned)blocks, kSerThreads, 0, s>>>(in, n, tok, s0, s1);
}

// Byte-grouped layout: a block takes kGrpTile consecutive groups of g bytes; each thread writes
// its groups' 2g digits and separator tokens into shared memory, and the block stores the tile's
// tokens as 16-byte vectors (a tile starts at token k0 (2g + ns), k0 a multiple of kGrpTile, so
// on a 16-byte boundary). Byte b of the stream is byte b mod 4 of fp32 value b / 4 (most
// significant first, or least with le) or uint8 code b.
constexpr int kGrpThreads = 256, kGrpTile = 4 * kGrpThreads;

__global__ void __launch_bounds__(kGrpThreads) k_serialize_grouped(const void* __restrict__ in, int64_t n, int bv,
                                                                   int g, int ns, int le,
                                                                   uint16_t* __restrict__ tok, uint16_t sep0,
                                                                   uint16_t sep1, bool vec) {
  __shared__ __align__(16) uint16_t buf[kGrpTile * (2 * 8 + 2)];
  const int64_t nb = n * bv, n_groups = (nb + g - 1) / g;
  const int64_t k0 = (int64_t)blockIdx.x * kGrpTile;
  const int tpg = 2 * g + ns;
  const int ng = n_groups - k0 < kGrpTile ? (int)(n_groups - k0) : kGrpTile;
  for (int i = threadIdx.x; i < ng; i += kGrpThreads) {
    const int64_t b0 = (k0 + i) * g, b1 = b0 + g < nb ? b0 + g : nb;
    uint16_t* o = buf + i * tpg;
    for (int64_t b = b0; b < b1; b++) {
      uint32_t byte;
      if (bv == 1) {
        byte = reinterpret_cast<const uint8_t*>(in)[b];
      } else {
        const int j = (int)(b & 3);
        byte = (reinterpret_cast<const uint32_t*>(in)[b >> 2] >> (le ? 8 * j : 8 * (3 - j))) & 0xFFu;
      }
      *o++ = (uint16_t)(byte >> 4);
      *o++ = (uint16_t)(byte & 0xFu);
    }
    if (ns >= 1) *o++ = sep0;
    if (ns >= 2) *o = sep1;
  }
  __syncthreads();
  // the tile's tokens (the last group of the stream may be short)
  const int64_t t0 = k0 * tpg;
  const int64_t tend = 2 * nb + (int64_t)ns * n_groups;
  const int nt = tend - t0 < (int64_t)kGrpTile * tpg ? (int)(tend - t0) : kGrpTile * tpg;
  uint16_t* dst = tok + t0;
  if (vec) {
    const uint4* s4 = reinterpret_cast<const uint4*>(buf);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (int q = threadIdx.x; q < nt / 8; q += kGrpThreads) __stcs(d4 + q, s4[q]);
    for (int q = (nt / 8) * 8 + threadIdx.x; q < nt; q += kGrpThreads) dst[q] = buf[q];
  } else {
    for (int q = threadIdx.x; q < nt; q += kGrpThreads) dst[q] = buf[q];
  }
}

void launch_serialize(int input_kind, int sep_mode, int byte_group, int byte_order, const void* in, int64_t n,
                      uint16_t* tok, cudaStream_t s) {
  if (n <= 0) return;
  note_launch();
  uint16_t s0, s1;
  sep_ids(sep_mode, &s0, &s1);
  if (!serial_is_default(input_kind, byte_group, byte_order)) {
    const int bv = (int)bytes_per_value(input_kind), g = byte_group ? byte_group : bv;
    const int64_t groups = (n * bv + g - 1) / g;
    const bool vec = ((uintptr_t)tok) % 16 == 0;  // tiles start on 16-byte boundaries then
    k_serialize_grouped<<<(unsigned)((groups + kGrpTile - 1) / kGrpTile), kGrpThreads, 0, s>>>(
        in, n, bv, g, sep_count(sep_mode), byte_order, tok, s0, s1, vec);
    return;
  }
  int ns = sep_mode == LMGC_SEP_NONE ? 0 : (sep_mode == LMGC_SEP_COMMA_SPACE ? 2 : 1);
  bool vec = (((uintptr_t)in) % 16 == 0) && (((uintptr_t)tok) % 16 == 0);
  if (input_kind == LMGC_IN_F32) {
    if (ns == 0) ser_dispatch<8, 0>(vec, in, n, tok, s0, s1, s);
    else if (ns == 1) ser_dispatch<8, 1>(vec, in, n, tok, s0, s1, s);
    else ser_dispatch<8, 2>(vec, in, n, tok, s0, s1, s);
  } else {
    if (ns == 0) ser_dispatch<2, 0>(vec, in, n, tok, s0, s1, s);
    else if (ns == 1) ser_dispatch<2, 1>(vec, in, n, tok, s0, s1, s);
    else ser_dispatch<2, 2>(vec, in, n, tok, s0, s1, s);
  }
}

// Inverse: one thread per value; a malformed group sets kErrDeser in *err.
__global__ void k_deserialize(const uint16_t* __restrict__ tok, int64_t n, int nd, int ns, uint16_t sep0,
                              uint16_t sep1, void* __restrict__ out, uint32_t* err) {
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int tpv = nd + ns;
  const uint16_t* g = tok + i * tpv;
  uint32_t b = 0;
  bool bad = false;
  for (int j = 0; j < nd; j++) {
    uint16_t d = g[j];
    bad |= d > 15;
    b = (b << 4) | (d & 0xFu);
  }
  if (ns >= 1) bad |= g[nd] != sep0;
  if (ns >= 2) bad |= g[nd + 1] != sep1;
  if (bad) atomicOr(err, kErrDeser);
  if (nd == 8) reinterpret_cast<uint32_t*>(out)[i] = b;
  else reinterpret_cast<uint8_t*>(out)[i] = (uint8_t)b;
}

// Inverse of k_serialize_grouped: one thread per group; each byte lands at its place in the
// output (fp32 values are little-endian in memory); a malformed group sets kErrDeser.
__global__ void k_deserialize_grouped(const uint16_t* __restrict__ tok, int64_t n, int bv, int g, int ns, int le,
                                      uint16_t sep0, uint16_t sep1, uint8_t* __restrict__ out, uint32_t* err) {
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t nb = n * bv;
  if (k >= (nb + g - 1) / g) return;
  const int64_t b0 = k * g, b1 = b0 + g < nb ? b0 + g : nb;
  const uint16_t* t = tok + 2 * b0 + ns * k;
  bool bad = false;
  for (int64_t b = b0; b < b1; b++) {
    const uint16_t hi = *t++, lo = *t++;
    bad |= hi > 15 || lo > 15;
    const uint8_t byte = (uint8_t)(((hi & 0xFu) << 4) | (lo & 0xFu));
    if (bv == 1) {
      out[b] = byte;
    } else {
      const int j = (int)(b & 3), shift = le ? 8 * j : 8 * (3 - j);
      out[(b >> 2) * 4 + shift / 8] = byte;
    }
  }
  if (ns >= 1) bad |= *t++ != sep0;
  if (ns >= 2) bad |= *t != sep1;
  if (bad) atomicOr(err, kErrDeser);
}

void launch_deserialize(int input_kind, int sep_mode, int byte_group, int byte_order, const uint16_t* tok,
                        int64_t n_values, void* out, uint32_t* err, cudaStream_t s) {
  if (n_values <= 0) return;
  uint16_t s0, s1;
  sep_ids(sep_mode, &s0, &s1);
  if (!serial_is_default(input_kind, byte_group, byte_order)) {
    const int bv = (int)bytes_per_value(input_kind), g = byte_group ? byte_group : bv;
    const int64_t groups = (n_values * bv + g - 1) / g;
    note_launch();
    k_deserialize_grouped<<<(unsigned)((groups + 255) / 256), 256, 0, s>>>(
        tok, n_values, bv, g, sep_count(sep_mode), byte_order, s0, s1, reinterpret_cast<uint8_t*>(out), err);
    return;
  }
  int ns = sep_mode == LMGC_SEP_NONE ? 0 : (sep_mode == LMGC_SEP_COMMA_SPACE ? 2 : 1);
  int nd = input_kind == LMGC_IN_F32 ? 8 : 2;
  note_launch();
  k_deserialize<<<(unsigned)((n_values + 255) / 256), 256, 0, s>>>(tok, n_values, nd, ns, s0, s1, out, err);
}

}  // namespace lmgc
