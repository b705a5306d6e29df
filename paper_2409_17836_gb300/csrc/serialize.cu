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

// Byte-grouped layout. Byte b of the stream is byte b mod 4 of fp32 value b / 4 (most
// significant first, or least with le) or uint8 code b. Tokens of group k start at k (2g + ns).
//
// k_serialize_units (whole tiles of a word-aligned stream): a thread takes one unit of lcm(g, 4)
// bytes -- whole words, lcm(g, 4) / g whole groups -- loads its words, writes the unit's digit and
// separator tokens into shared memory, and the block stores the tile's tokens as 16-byte vectors.
// k_serialize_grouped (the rest, from group k_base): a block takes kGrpTile consecutive groups,
// a thread a group at a time, bytes loaded one by one (it also takes the stream's short last
// group). Both tiles start on 16-byte boundaries of the token array (their first group is a
// multiple of 256 groups), and the shared tile is sized for the launch's g and ns.
constexpr int kGrpThreads = 256, kGrpTile = 4 * kGrpThreads;

template <int G>
struct GroupUnit {
  static constexpr int kBytes = G % 4 == 0 ? G : (G % 2 == 0 ? 2 * G : 4 * G);  // lcm(G, 4)
  static constexpr int kWords = kBytes / 4;
  static constexpr int kGroups = kBytes / G;
};

template <int G>
__global__ void __launch_bounds__(kGrpThreads, 8) k_serialize_units(const uint32_t* __restrict__ in, int ns,
                                                                 int swap, uint16_t* __restrict__ tok,
                                                                 uint16_t sep0, uint16_t sep1) {
  using U = GroupUnit<G>;
  extern __shared__ __align__(16) uint16_t ubuf[];  // kGrpThreads * U::kGroups * (2 G + ns) tokens
  const int tpg = 2 * G + ns, ut = U::kGroups * tpg;
  const int t = threadIdx.x;
  const uint32_t* src = in + ((int64_t)blockIdx.x * kGrpThreads + t) * U::kWords;
  uint32_t w[U::kWords];
#pragma unroll
  for (int i = 0; i < U::kWords; i++) {
    w[i] = __ldcs(src + i);
    if (swap) w[i] = __byte_perm(w[i], 0u, 0x0123);  // most significant byte first: byte j at bits 8j
  }
  uint16_t* o = ubuf + t * ut;
#pragma unroll
  for (int k = 0; k < U::kGroups; k++) {
#pragma unroll
    for (int i = 0; i < G; i++) {
      const int b = k * G + i;  // the unit's byte b: byte b & 3 of word b >> 2
      const uint32_t byte = (w[b >> 2] >> (8 * (b & 3))) & 0xFFu;
      o[2 * i] = (uint16_t)(byte >> 4);
      o[2 * i + 1] = (uint16_t)(byte & 0xFu);
    }
    if (ns >= 1) o[2 * G] = sep0;
    if (ns >= 2) o[2 * G + 1] = sep1;
    o += tpg;
  }
  __syncthreads();
  const int nt = kGrpThreads * ut;  // a multiple of 8
  const uint4* s4 = reinterpret_cast<const uint4*>(ubuf);
  uint4* d4 = reinterpret_cast<uint4*>(tok + (int64_t)blockIdx.x * nt);
  for (int q = t; q < nt / 8; q += kGrpThreads) __stcs(d4 + q, s4[q]);
}

__global__ void __launch_bounds__(kGrpThreads) k_serialize_grouped(const void* __restrict__ in, int64_t n, int bv,
                                                                   int g, int ns, int le, int64_t k_base,
                                                                   uint16_t* __restrict__ tok, uint16_t sep0,
                                                                   uint16_t sep1, bool vec) {
  extern __shared__ __align__(16) uint16_t buf[];  // kGrpTile * (2 g + ns) tokens
  const int64_t nb = n * bv, n_groups = (nb + g - 1) / g;
  const int64_t k0 = k_base + (int64_t)blockIdx.x * kGrpTile;
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
    const int ns = sep_count(sep_mode);
    const int64_t nb = n * bv;
    // whole tiles of units (word loads need a word-aligned stream; the tile stores 16-byte ones)
    int64_t k_base = 0;
    if (vec && (bv == 4 || ((uintptr_t)in) % 4 == 0)) {
      const int swap = bv == 4 && !byte_order;  // fp32 bytes most significant first
      const uint32_t* w = reinterpret_cast<const uint32_t*>(in);
#define LMGC_UNITS(GV)                                                                                          \
  do {                                                                                                           \
    using U = GroupUnit<GV>;                                                                                     \
    const int64_t tiles = nb / ((int64_t)kGrpThreads * U::kBytes);                                               \
    if (tiles > 0) {                                                                                             \
      const size_t sm = (size_t)kGrpThreads * U::kGroups * (size_t)(2 * GV + ns) * sizeof(uint16_t);            \
      k_serialize_units<GV><<<(unsigned)tiles, kGrpThreads, sm, s>>>(w, ns, swap, tok, s0, s1);                 \
      k_base = tiles * kGrpThreads * U::kGroups;                                                                  \
    }                                                                                                            \
  } while (0)
      switch (g) {
        case 1: LMGC_UNITS(1); break;
        case 2: LMGC_UNITS(2); break;
        case 3: LMGC_UNITS(3); break;
        case 4: LMGC_UNITS(4); break;
        case 5: LMGC_UNITS(5); break;
        case 6: LMGC_UNITS(6); break;
        case 7: LMGC_UNITS(7); break;
        default: LMGC_UNITS(8); break;
      }
#undef LMGC_UNITS
    }
    if (k_base < groups) {
      if (k_base > 0) note_launch();
      const size_t smem = (size_t)kGrpTile * (size_t)(2 * g + ns) * sizeof(uint16_t);  // <= 36 KB (g <= 8)
      k_serialize_grouped<<<(unsigned)((groups - k_base + kGrpTile - 1) / kGrpTile), kGrpThreads, smem, s>>>(
          in, n, bv, g, ns, byte_order, k_base, tok, s0, s1, vec);
    }
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
