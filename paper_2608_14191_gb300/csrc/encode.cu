// AATC encode on sm_103a (Algorithm 1 "Project" + "Append qtz(h)"; quantizer of Sec. 5).
//
// aatc_encode_kernel: one persistent CTA per (basis, slice of work): a basis is one (layer,
// kv-head, K|V) stream, an item is 128 consecutive new tokens of one sequence.  Warp roles:
//   warp 12   : TMA producer -- 128 x 128 bf16 token tiles into a 5-stage SW128 ring,
//   warp 13   : MMA issuer   -- tcgen05.mma (M=128 tokens, N=128 channels, K=128) into one of
//                               four TMEM accumulators (all 512 columns; item i -> accumulator i % 4),
//   warps 0-11: three epilogue warpgroups; group e drains items e, e+3, ...: thread = token =
//               TMEM lane: token scale alpha, quantize, and the packed record built from the
//               token's stored values held in registers (128 registers a thread: four of the
//               14 warps share a scheduler's 16 K registers).
// aatc_encode_hidden_kernel (further down) computes the coefficients from the layer input.
// The projection uses the plan's bf16 basis; accumulation is fp32.
#include <cudaTypedefs.h>
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <type_traits>

#include "aatc_internal.h"
#include "ptx.cuh"

namespace aatc {
namespace {

constexpr int kTileBytes = TILE * D * 2;          // 32 KB of bf16
constexpr int kEpiGroups = 4;
constexpr int kEpiThreads = 128 * kEpiGroups;
constexpr int kProducerWarp = kEpiThreads / 32;
constexpr int kMmaWarp = kProducerWarp + 1;
constexpr int kThreads = kEpiThreads + 64;
constexpr int kAccCols = 128;                     // fp32 columns per accumulator
constexpr uint32_t kTmemCols = 512;               // four accumulators
constexpr int kByteRow = 132;                     // padded per-thread row of stored values

struct EncodeArgs {
  const ChanEnc* enc;     // plan tables (whole plan)
  const float* inv_s;
  const StreamLayout* lay;
  const short* entry;
  int* err;
  uint32_t* words;        // cache word region (this layer)
  float* alpha;           // cache alpha region
  int layer, n_kv, batch, start, n_tokens, n_chunks, n_words, n_tiles, n_entries, ctas_per_basis;
};

template <typename Smem>
__device__ __forceinline__ void raise_abort(Smem& sm, int* err) {
  sm.abort_flag = 1;
  atomicOr(err, 2);
}

// Writes one finished record word of a token.  Keys: plain word-planar store.  Values: the four
// byte-quarters go to the token's byte of the four slots of its 4-token block (slot positions
// 0, 2, 1, 3 for quarters 0..3), so each token only writes its own bytes.
struct RecordWriter {
  uint32_t* key_word;     // keys: &words[.. tile][0][lane]
  uint8_t* val_byte;      // values: byte (token % 4) of slot 4 (token / 4), record word 0
  bool value;
  __device__ __forceinline__ void put(int wi, uint32_t w) const {
    if (!value) {
      key_word[static_cast<size_t>(wi) * TILE] = w;
    } else {
      uint8_t* p = val_byte + static_cast<size_t>(wi) * TILE * 4;
      p[0] = static_cast<uint8_t>(w);
      p[8] = static_cast<uint8_t>(w >> 8);
      p[4] = static_cast<uint8_t>(w >> 16);
      p[12] = static_cast<uint8_t>(w >> 24);
    }
  }
};


// Token scale and stored values of one token (thread = token = TMEM lane): alpha = max over
// retained channels of |h_c| / s_c (inv_s = 0 for dropped ones), then u_c = clamp(floor(h_c /
// Delta_c + 1/2)) + 2^(b_c - 1) with Delta_c = alpha f_c, one byte per channel into `row`.  The
// 128 coefficients are read from TMEM columns taddr .. taddr + 127 (twice: amax, then quantize).
__device__ __forceinline__ float quantize_token(uint32_t taddr, const ChanEnc* enc, const float* inv_s,
                                                uint32_t* row) {
  // Eight 32-column TMEM loads (four per pass), each issued before the previous chunk is
  // processed so its latency overlaps that work; registers alternate between ra and rb.
  uint32_t ra[32], rb[32];
  float amax = 0.0f;
  auto amax_chunk = [&](const uint32_t (&r)[32], int j) {
#pragma unroll
    for (int i = 0; i < 32; i += 4) {
      const float4 is = *reinterpret_cast<const float4*>(&inv_s[32 * j + i]);
      amax = fmaxf(amax, fabsf(__uint_as_float(r[i])) * is.x);
      amax = fmaxf(amax, fabsf(__uint_as_float(r[i + 1])) * is.y);
      amax = fmaxf(amax, fabsf(__uint_as_float(r[i + 2])) * is.z);
      amax = fmaxf(amax, fabsf(__uint_as_float(r[i + 3])) * is.w);
    }
  };
  float ia = 0.0f;
  // The round-down add of 1.5 2^23 + 2^(b-1) leaves u (< 256) in the low byte of the float.
  auto quant_chunk = [&](const uint32_t (&r)[32], int j) {
    uint32_t y[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const ChanEnc e = enc[32 * j + i];
      float x = fmaf(__uint_as_float(r[i]), e.inv_f * ia, 0.5f);   // h / Delta + 1/2
      x = fminf(x, e.hi);                                       // |h| / Delta <= 2^(b-1): only the top clamps
      y[i] = __float_as_uint(__fadd_rd(x, e.magic));            // floor, offset binary in the mantissa
    }
#pragma unroll
    for (int q = 0; q < 8; ++q)
      row[8 * j + q] = __byte_perm(__byte_perm(y[4 * q], y[4 * q + 1], 0x0040),
                                   __byte_perm(y[4 * q + 2], y[4 * q + 3], 0x0040), 0x5410);
  };
  ptx::tmem_ld_32raw(taddr, ra);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  amax_chunk(ra, 0);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  amax_chunk(rb, 1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  amax_chunk(ra, 2);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr, ra);
  amax_chunk(rb, 3);
  ia = amax > 0.0f ? 1.0f / amax : 0.0f;
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  quant_chunk(ra, 0);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  quant_chunk(rb, 1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  quant_chunk(ra, 2);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  quant_chunk(rb, 3);
  return amax;
}

// 16 base-4 digits (bits sh, sh + 1 of the bytes of channels 4q .. 4q + 15) as one 32-bit chunk,
// channel order LSB first.  Per row word, mask and multiply drop its four digits into the top
// byte: digit i sits at bit 8i + sh, the multiplier terms 2^(24 - sh - 6j) move it to 24 + 2i
// (j = i); every cross term lands below bit 24 at its own position or above bit 31, so no carry
// reaches the top byte.
__device__ __forceinline__ uint32_t gather_d2(const uint32_t* row, int q, int sh) {
  const uint32_t m = 0x03030303u << sh, mul = 0x01041040u >> sh;
  uint32_t p[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) p[i] = (row[min(q + i, 31)] & m) * mul;
  return __byte_perm(__byte_perm(p[0], p[1], 0x0073), __byte_perm(p[2], p[3], 0x0073), 0x5410);
}
// 32 single bits (bit sh of channels 4q .. 4q + 31) as one chunk.  Two row words are merged
// first (the second one's bits 4 higher), then multiplier terms 2^(24 - s - 7j) move bit i of the
// first word to 24 + i and of the second to 28 + i: eight channels per top byte.
__device__ __forceinline__ uint32_t gather_d1(const uint32_t* row, int q, int sh) {
  const int pre = sh >= 4 ? 4 : 0, s = sh - pre;        // the multiplier needs s <= 3
  const uint32_t m = 0x01010101u << s, mul = 0x01020408u >> s;
  uint32_t p[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t x0 = row[min(q + 2 * i, 31)] >> pre, x1 = row[min(q + 2 * i + 1, 31)] >> pre;
    p[i] = ((x0 & m) | ((x1 << 4) & (m << 4))) * mul;
  }
  return __byte_perm(__byte_perm(p[0], p[1], 0x0073), __byte_perm(p[2], p[3], 0x0073), 0x5410);
}

// Packed record of one token from its byte row: the bit stream of Sec. 5's stored values in the
// D2 / D1 layout (field w bits at bit sh of channels [c0, c1), w = 2: a base-4 digit, w = 1: a
// single bit), appended LSB first in 32-bit chunks.
__device__ __forceinline__ void pack_token(const StreamLayout& lay, const uint32_t* row, const RecordWriter& out,
                                           int n_words) {
  uint32_t word = 0;
  int pos = 0, wi = 0;                                  // uniform across the warp: same layout
  auto append = [&](uint32_t v, int nb) {               // v: nb (1 .. 32) valid bits, zero above
    word |= v << pos;
    if (pos + nb >= 32) {
      out.put(wi, word);
      ++wi;
      word = __funnelshift_rc(v, 0u, 32 - pos);         // the bits that did not fit (none at pos 0)
    }
    pos = (pos + nb) & 31;
  };
  auto emit_run = [&](int c0, int c1, int sh, int w) {
    int drop = w * (c0 & 3);                            // chunks start on row words
    for (int cb = c0 & ~3; cb < c1; cb += 32 / w) {
      uint32_t v = w == 2 ? gather_d2(row, cb >> 2, sh) : gather_d1(row, cb >> 2, sh);
      int nb = min(w * (c1 - cb), 32);
      if (nb < 32) v &= (1u << nb) - 1u;
      v >>= drop;
      nb -= drop;
      drop = 0;
      append(v, nb);
    }
  };
#pragma unroll
  for (int k = 0; k < 4; ++k) emit_run(0, lay.l2[k], 2 * k, 2);                 // D2 digits
#pragma unroll
  for (int k = 3; k >= 0; --k) emit_run(lay.l2all[k], lay.lodd[k], 2 * k, 1);  // D1: top bits of odd widths
#pragma unroll
  for (int k = 0; k < 4; ++k) emit_run(lay.l2[k], lay.l2all[k], 2 * k, 2);     // D1: digits moved out of D2
  if (pos > 0) {
    out.put(wi, word);
    ++wi;
  }
  for (; wi < n_words; ++wi) out.put(wi, 0u);
}

// Writer for token position pos_t of cache stream sidx.
__device__ __forceinline__ RecordWriter record_writer(uint32_t* words, size_t sidx, size_t stream_words,
                                                      int n_words, int pos_t, bool value) {
  uint32_t* tile_words = words + sidx * stream_words + static_cast<size_t>(pos_t / TILE) * n_words * TILE;
  RecordWriter out;
  out.value = value;
  const int tt = pos_t % TILE;
  out.key_word = tile_words + tt;
  out.val_byte = reinterpret_cast<uint8_t*>(tile_words + 4 * (tt >> 2)) + (tt & 3);
  return out;
}

// ------------------------------------------------------------------ register-resident epilogue
constexpr int kKStages = 5;                       // input stages of aatc_encode_kernel
constexpr int kKGroups = 3;                       // epilogue warpgroups
constexpr int kKAcc = 4;                          // TMEM accumulators
constexpr int kKEpiThreads = 128 * kKGroups;
constexpr int kKProducerWarp = kKEpiThreads / 32;
constexpr int kKMmaWarp = kKProducerWarp + 1;
constexpr int kKThreads = kKEpiThreads + 64;

struct QuantTables {      // per channel, structure of arrays (16-byte aligned)
  const float* inv_s;     // 1 / s_c (0 for dropped channels)
  const float* inv_f;     // 1 / f_c
  const float* hi;        // upper clamp of h / Delta + 1/2
  const float* magic;     // 1.5 2^23 + 2^(b_c - 1)
};

// alpha pass over 32 channels (TMEM columns 32 j ..): running maxima of |h_c| / s_c, two per
// instruction (inv_s = 0 for dropped channels).
__device__ __forceinline__ void amax_chunk_regs(const uint32_t (&r)[32], int j, const float* inv_s, float& am0,
                                                float& am1) {
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 is = ptx::lds_f4(&inv_s[32 * j + i]);
    float a0, a1, a2, a3;
    ptx::f2_unpack(ptx::f2_mul(ptx::f2_pack(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), ptx::f2_pack(is.x, is.y)),
                   a0, a1);
    ptx::f2_unpack(ptx::f2_mul(ptx::f2_pack(__uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])), ptx::f2_pack(is.z, is.w)),
                   a2, a3);
    am0 = ptx::fmax3(am0, fabsf(a0), fabsf(a1));
    am1 = ptx::fmax3(am1, fabsf(a2), fabsf(a3));
  }
}
// quantize pass over 32 channels: x = h / Delta + 1/2 = h (ia / f_c) + 1/2, clamped above, then
// the round-down add of 1.5 2^23 + 2^(b-1) leaves u (< 2^16) in the low two bytes of the float;
// U gets the low bytes of channels 32 j .., UH (kWide, j = 0 only) the high bytes.
template <bool kWide>
__device__ __forceinline__ void quant_chunk_regs(const uint32_t (&r)[32], int j, const QuantTables& tb, uint64_t ia2,
                                                 uint32_t (&U)[32], uint32_t (&UH)[8]) {
  const uint64_t half2 = ptx::f2_pack(0.5f, 0.5f);
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 f = ptx::lds_f4(&tb.inv_f[32 * j + i]);
    const float4 h = ptx::lds_f4(&tb.hi[32 * j + i]);
    const float4 m = ptx::lds_f4(&tb.magic[32 * j + i]);
    float x0, x1, x2, x3;
    ptx::f2_unpack(ptx::f2_fma(ptx::f2_pack(__uint_as_float(r[i]), __uint_as_float(r[i + 1])),
                               ptx::f2_mul(ptx::f2_pack(f.x, f.y), ia2), half2), x0, x1);
    ptx::f2_unpack(ptx::f2_fma(ptx::f2_pack(__uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])),
                               ptx::f2_mul(ptx::f2_pack(f.z, f.w), ia2), half2), x2, x3);
    float y0, y1, y2, y3;
    ptx::f2_unpack(ptx::f2_add_rd(ptx::f2_pack(fminf(x0, h.x), fminf(x1, h.y)), ptx::f2_pack(m.x, m.y)), y0, y1);
    ptx::f2_unpack(ptx::f2_add_rd(ptx::f2_pack(fminf(x2, h.z), fminf(x3, h.w)), ptx::f2_pack(m.z, m.w)), y2, y3);
    U[8 * j + i / 4] = __byte_perm(__byte_perm(__float_as_uint(y0), __float_as_uint(y1), 0x0040),
                                   __byte_perm(__float_as_uint(y2), __float_as_uint(y3), 0x0040), 0x5410);
    if (kWide && j == 0)
      UH[i / 4] = __byte_perm(__byte_perm(__float_as_uint(y0), __float_as_uint(y1), 0x0051),
                              __byte_perm(__float_as_uint(y2), __float_as_uint(y3), 0x0051), 0x5410);
  }
}

// Token scale and stored values of one token (thread = token = TMEM lane), as quantize_token
// but two channels per fp32 instruction and the stored values kept in registers: U[w] holds the
// low bytes of u_c for channels 4w .. 4w + 3, UH[w] the high bytes (u_c >= 256 only for widths
// above 8, which lie in the first 32 channels).  The arithmetic (and so every code) is the same.
// Eight 32-column TMEM loads (four per pass), each issued before the previous chunk is processed
// so its latency overlaps that work.
template <bool kWide>
__device__ __forceinline__ float quantize_token_regs(uint32_t taddr, const QuantTables& tb, uint32_t (&U)[32],
                                                     uint32_t (&UH)[8]) {
  uint32_t ra[32], rb[32];
  float am0 = 0.0f, am1 = 0.0f;
  ptx::tmem_ld_32raw(taddr, ra);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  amax_chunk_regs(ra, 0, tb.inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  amax_chunk_regs(rb, 1, tb.inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  amax_chunk_regs(ra, 2, tb.inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr, ra);
  amax_chunk_regs(rb, 3, tb.inv_s, am0, am1);
  const float amax = fmaxf(am0, am1);
  const float ia = amax > 0.0f ? 1.0f / amax : 0.0f;
  const uint64_t ia2 = ptx::f2_pack(ia, ia);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  quant_chunk_regs<kWide>(ra, 0, tb, ia2, U, UH);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  quant_chunk_regs<kWide>(rb, 1, tb, ia2, U, UH);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  quant_chunk_regs<kWide>(ra, 2, tb, ia2, U, UH);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  quant_chunk_regs<kWide>(rb, 3, tb, ia2, U, UH);
  return amax;
}

// The two passes separately, for head-group streams whose alpha spans several slices: the
// slice's maximum of |h_c| / s_c, then its stored values for a given 1 / alpha.
__device__ __forceinline__ float token_amax_regs(uint32_t taddr, const float* inv_s) {
  uint32_t ra[32], rb[32];
  float am0 = 0.0f, am1 = 0.0f;
  ptx::tmem_ld_32raw(taddr, ra);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  amax_chunk_regs(ra, 0, inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  amax_chunk_regs(rb, 1, inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  amax_chunk_regs(ra, 2, inv_s, am0, am1);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  amax_chunk_regs(rb, 3, inv_s, am0, am1);
  return fmaxf(am0, am1);
}
__device__ __forceinline__ void token_quant_regs(uint32_t taddr, const QuantTables& tb, float ia, uint32_t (&U)[32]) {
  uint32_t ra[32], rb[32], uh[8];
  const uint64_t ia2 = ptx::f2_pack(ia, ia);
  ptx::tmem_ld_32raw(taddr, ra);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 32, rb);
  quant_chunk_regs<false>(ra, 0, tb, ia2, U, uh);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  ptx::tmem_ld_32raw(taddr + 64, ra);
  quant_chunk_regs<false>(rb, 1, tb, ia2, U, uh);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(ra);
  ptx::tmem_ld_32raw(taddr + 96, rb);
  quant_chunk_regs<false>(ra, 2, tb, ia2, U, uh);
  ptx::tmem_ld_wait();
  ptx::tmem_regs_ready(rb);
  quant_chunk_regs<false>(rb, 3, tb, ia2, U, uh);
}

// Base-4 digit k of the 16 channels held in w0 .. w3, channel order LSB first: the mask-and-
// multiply of gather_d2 on registers (m = 0x03030303 << 2k, mul = 0x01041040 >> 2k).
__device__ __forceinline__ uint32_t digits16(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3, uint32_t m,
                                             uint32_t mul) {
  return __byte_perm(__byte_perm((w0 & m) * mul, (w1 & m) * mul, 0x0073),
                     __byte_perm((w2 & m) * mul, (w3 & m) * mul, 0x0073), 0x5410);
}
// Bit sh = pre + s (s <= 3) of the 8 channels held in w0, w1 as the top byte (gather_d1's merge
// and multiply: m = 0x01010101 << s, mul = 0x01020408 >> s).
__device__ __forceinline__ uint32_t bits8_top(uint32_t w0, uint32_t w1, int pre, uint32_t m, uint32_t mul) {
  return (((w0 >> pre) & m) | (((w1 >> pre) << 4) & (m << 4))) * mul;
}
// That bit of the 32 channels held in U[8i] .. U[8i + 7], channel order LSB first.
template <int N>
__device__ __forceinline__ uint32_t bits32(const uint32_t (&U)[N], int i, int pre, uint32_t m, uint32_t mul) {
  return __byte_perm(__byte_perm(bits8_top(U[8 * i], U[8 * i + 1], pre, m, mul),
                                 bits8_top(U[8 * i + 2], U[8 * i + 3], pre, m, mul), 0x0073),
                     __byte_perm(bits8_top(U[8 * i + 4], U[8 * i + 5], pre, m, mul),
                                 bits8_top(U[8 * i + 6], U[8 * i + 7], pre, m, mul), 0x0073),
                     0x5410);
}

// Writes one token's record words in order.  Keys: word-planar, token lane t of a tile in column
// t of each record word.  Values: tokens 4Q .. 4Q+3 share slots 4Q .. 4Q+3 of each record word,
// slot 4Q + (0, 2, 1, 3)[r] holding byte-quarter r of the four tokens' words (token 4Q + i in
// byte i): each token writes its own four bytes.  (Whole slot words through a byte transpose
// across the lane quad measured slower: the larger inlined flush lengthened the code executed per
// record word, which a kernel started after other work fetches from memory.)
struct RecordFlush {
  uint32_t* tile_words;   // record word 0 of the token's tile
  int tt;                 // token lane inside the tile
  bool value, ok;
  int wi;
  __device__ __forceinline__ void operator()(uint32_t w) {
    uint32_t* rw = tile_words + static_cast<size_t>(wi) * TILE;
    if (ok) {
      if (!value) {
        rw[tt] = w;
      } else {
        uint8_t* q = reinterpret_cast<uint8_t*>(rw + 4 * (tt >> 2)) + (tt & 3);
        q[0] = static_cast<uint8_t>(w);
        q[8] = static_cast<uint8_t>(w >> 8);
        q[4] = static_cast<uint8_t>(w >> 16);
        q[12] = static_cast<uint8_t>(w >> 24);
      }
    }
    ++wi;
  }
};

// The packed record of one token from its stored values in registers, in the layout of
// pack_token: D2 digits layer by layer (the last n2 % 16 of them moved behind the D1 top bits),
// the top bit of every odd-width channel, the moved digits, zeros up to n_words.  Digit layers
// and bit positions run as loops; the channel chunks inside them are unrolled (registers are
// indexed at compile time) and guarded by the stream's run bounds, which are the same for every
// thread of the CTA.  Digit layers 4..7 and the top bits of widths 9..15 come from the high
// bytes UH (channels 0..31).
template <bool kWide>
__device__ __forceinline__ void pack_token_regs(const StreamLayout& lay, const uint32_t (&U)[32],
                                                const uint32_t (&UH)[8], RecordFlush& flush, int n_words) {
  uint32_t word = 0;
  int pos = 0;
  auto put = [&](uint32_t v, int nb) {                   // v: nb (1 .. 32) valid bits, zero above
    word |= v << pos;
    if (pos + nb >= 32) {
      flush(word);
      word = __funnelshift_rc(v, 0u, 32 - pos);           // the bits that did not fit (none at pos 0)
    }
    pos = (pos + nb) & 31;
  };
  uint32_t moved = 0;
  int mpos = 0;
  // chunk c (channels 16c .. 16c + 15) of a digit layer whose run is [0, la), the first lk kept
  auto digit_chunk = [&](uint32_t v, int c, int lk, int la) {
    if (16 * c + 16 <= lk) {                               // the whole chunk stays in D2
      put(v, 32);
      return;
    }
    const int nm = max(lk - 16 * c, 0);                    // digits that stay in D2 (< 16)
    const int nt = min(la - 16 * c, 16);                   // digits of this chunk
    if (nm > 0) put(v & ((1u << (2 * nm)) - 1u), 2 * nm);
    if (nt > nm) {                                         // at most 15 digits move in all
      moved |= (__funnelshift_rc(v, 0u, 2 * nm) & ((1u << (2 * (nt - nm))) - 1u)) << mpos;
      mpos += 2 * (nt - nm);
    }
  };
#pragma unroll 1
  for (int k = 0; k < (kWide ? 8 : 4); ++k) {
    const int lk = lay.l2[k], la = lay.l2all[k];          // non-increasing in k
    if (la == 0) break;
    const uint32_t m = 0x03030303u << (2 * (k & 3)), mul = 0x01041040u >> (2 * (k & 3));
    if (!kWide || k < 4) {
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        if (16 * c >= la) break;
        digit_chunk(digits16(U[4 * c], U[4 * c + 1], U[4 * c + 2], U[4 * c + 3], m, mul), c, lk, la);
      }
    } else {                                               // la <= 32: widths above 8
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        if (16 * c >= la) break;
        digit_chunk(digits16(UH[4 * c], UH[4 * c + 1], UH[4 * c + 2], UH[4 * c + 3], m, mul), c, lk, la);
      }
    }
  }
#pragma unroll 1
  for (int k = kWide ? 7 : 3; k >= 0; --k) {
    const int a = lay.l2all[k], b = lay.lodd[k];          // width 2k + 1 channels [a, b)
    if (a >= b) continue;
    const int pre = (k & 3) >= 2 ? 4 : 0, s = 2 * (k & 3) - pre;
    const uint32_t m = 0x01010101u << s, mul = 0x01020408u >> s;
    if (!kWide || k < 4) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (a < 32 * i + 32 && b > 32 * i) {
          const int lo = max(a - 32 * i, 0), n = min(b - 32 * i, 32) - lo;
          uint32_t v = __funnelshift_rc(bits32(U, i, pre, m, mul), 0u, lo);
          if (n < 32) v &= (1u << n) - 1u;
          put(v, n);
        }
      }
    } else {                                               // widths 9 .. 15: b <= 32
      const int n = b - a;
      uint32_t v = __funnelshift_rc(bits32(UH, 0, pre, m, mul), 0u, a);
      if (n < 32) v &= (1u << n) - 1u;
      put(v, n);
    }
  }
  if (mpos > 0) put(moved, mpos);
  if (pos > 0) flush(word);
  while (flush.wi < n_words) flush(0u);
}

struct EncodeSmem {
  alignas(1024) unsigned char u_tile[kTileBytes];
  alignas(1024) unsigned char x_tile[kKStages][kTileBytes];
  alignas(16) float inv_s[D];
  alignas(16) float inv_f[D];
  alignas(16) float hi[D];
  alignas(16) float magic[D];
  StreamLayout lay;
  uint64_t full[kKStages], empty[kKStages], tfull[kKAcc], tempty[kKAcc], ubar;
  uint32_t tmem_base;
  int abort_flag;
};

__global__ void __launch_bounds__(kKThreads, 1)
    aatc_encode_kernel(const __grid_constant__ CUtensorMap tmap_k, const __grid_constant__ CUtensorMap tmap_v,
                       const __grid_constant__ CUtensorMap tmap_u, const EncodeArgs a) {
  extern __shared__ unsigned char smem_raw[];
  EncodeSmem& sm = *reinterpret_cast<EncodeSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;

  const int basis = blockIdx.x / a.ctas_per_basis;           // (kv-head, kind) inside the layer
  const int sub = blockIdx.x % a.ctas_per_basis;
  const int head = basis >> 1, kind = basis & 1;
  const int stream = (a.layer * a.n_kv + head) * 2 + kind;
  const long n_items = static_cast<long>(a.batch) * a.n_chunks;
  const long it0 = n_items * sub / a.ctas_per_basis;
  const long it1 = n_items * (sub + 1) / a.ctas_per_basis;
  const int my_items = static_cast<int>(it1 - it0);
  const CUtensorMap* tmap_x = kind == 0 ? &tmap_k : &tmap_v;

  // per-stream tables
  for (int c = tid; c < D; c += kKThreads) {
    const ChanEnc e = a.enc[stream * D + c];
    sm.inv_s[c] = a.inv_s[stream * D + c];
    sm.inv_f[c] = e.inv_f;
    sm.hi[c] = e.hi;
    sm.magic[c] = e.magic;
  }
  if (tid == 0) {
    sm.lay = a.lay[stream];
    for (int s = 0; s < kKStages; ++s) {
      ptx::mbar_init(&sm.full[s], 1);
      ptx::mbar_init(&sm.empty[s], 1);
    }
    for (int j = 0; j < kKAcc; ++j) {
      ptx::mbar_init(&sm.tfull[j], 1);
      ptx::mbar_init(&sm.tempty[j], 128);
    }
    ptx::mbar_init(&sm.ubar, 1);
    sm.abort_flag = 0;
    ptx::fence_mbar_init();
  }
  if (warp == kKMmaWarp) {
    ptx::tmem_alloc(&sm.tmem_base, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == kKProducerWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && my_items > 0) {
      ptx::prefetch_tmap(tmap_x);
      ptx::prefetch_tmap(&tmap_u);
      ptx::mbar_arrive_expect_tx(&sm.ubar, kTileBytes);
      ptx::tma_load_2d(sm.u_tile, &tmap_u, &sm.ubar, 0, stream * D);
      ptx::tma_load_2d(sm.u_tile + kTileBytes / 2, &tmap_u, &sm.ubar, 64, stream * D);
      for (int it = 0; it < my_items; ++it) {
        const int s = it % kKStages;
        const uint32_t ph = (it / kKStages) & 1;
        if (!ptx::mbar_wait_bounded(&sm.empty[s], ph ^ 1, abort_flag)) { raise_abort(sm, a.err); break; }
        const long item = it0 + it;
        const int b = static_cast<int>(item / a.n_chunks);
        const int i0 = static_cast<int>(item % a.n_chunks) * TILE;
        ptx::mbar_arrive_expect_tx(&sm.full[s], kTileBytes);
        ptx::tma_load_4d(sm.x_tile[s], tmap_x, &sm.full[s], 0, head, i0, b);
        ptx::tma_load_4d(sm.x_tile[s] + kTileBytes / 2, tmap_x, &sm.full[s], 64, head, i0, b);
      }
    }
  } else if (warp == kKMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && my_items > 0) {
      constexpr uint32_t idesc = ptx::idesc_bf16_f32(128, 128);
      const uint32_t u_base = ptx::smem_u32(sm.u_tile);
      bool ok = ptx::mbar_wait_bounded(&sm.ubar, 0, abort_flag);
      if (!ok) raise_abort(sm, a.err);
      for (int it = 0; ok && it < my_items; ++it) {
        const int s = it % kKStages;
        const uint32_t ph = (it / kKStages) & 1;
        const int acc = it % kKAcc;
        const uint32_t aph = (it / kKAcc) & 1;
        if (!ptx::mbar_wait_bounded(&sm.tempty[acc], aph ^ 1, abort_flag)) { raise_abort(sm, a.err); break; }
        ptx::tc_fence_after();
        if (!ptx::mbar_wait_bounded(&sm.full[s], ph, abort_flag)) { raise_abort(sm, a.err); break; }
        ptx::tc_fence_after();
        const uint32_t x_base = ptx::smem_u32(sm.x_tile[s]);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t koff = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          ptx::umma_bf16(tmem + acc * kAccCols, ptx::sdesc_kmajor_sw128(x_base + koff),
                         ptx::sdesc_kmajor_sw128(u_base + koff), idesc, kk > 0 ? 1u : 0u);
        }
        ptx::umma_commit(&sm.empty[s]);
        ptx::umma_commit(&sm.tfull[acc]);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue: thread = token
    const int eg = warp >> 2;                                  // epilogue group
    const int quad = warp & 3;                                 // TMEM lane quadrant
    const int tl = quad * 32 + lane;                           // token lane inside the tile
    const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;
    const QuantTables tb{sm.inv_s, sm.inv_f, sm.hi, sm.magic};
    // one instantiation for streams with a channel wider than 8 bits (high bytes kept), one without
    auto drain = [&](auto wide_tag) {
      constexpr bool kWide = decltype(wide_tag)::value;
#pragma unroll 1
      for (int it = eg; it < my_items; it += kKGroups) {
        const int acc = it % kKAcc;
        const uint32_t aph = (it / kKAcc) & 1;
        if (!ptx::mbar_wait_bounded(&sm.tfull[acc], aph, abort_flag)) { raise_abort(sm, a.err); break; }
        ptx::tc_fence_after();
        const uint32_t taddr = tmem + acc * kAccCols + (static_cast<uint32_t>(quad * 32) << 16);
        uint32_t U[32], UH[8];
        const float amax = quantize_token_regs<kWide>(taddr, tb, U, UH);
        ptx::tc_fence_before();
        ptx::mbar_arrive(&sm.tempty[acc]);

        const long item = it0 + it;
        const int b = static_cast<int>(item / a.n_chunks);
        const int i = static_cast<int>(item % a.n_chunks) * TILE + tl;     // input token index
        const bool ok = i < a.n_tokens;
        if (!__any_sync(0xffffffffu, ok)) continue;
        const int pos_t = a.start + i;
        const size_t sidx = (static_cast<size_t>(b) * a.n_kv + head) * 2 + kind;
        if (ok) {
          if (!isfinite(amax)) atomicOr(a.err, 1);
          a.alpha[sidx * a.n_tiles * TILE + pos_t] = amax;
        }
        RecordFlush f{a.words + sidx * stream_words + static_cast<size_t>(pos_t / TILE) * a.n_words * TILE,
                      pos_t % TILE, kind == 1, ok, 0};
        pack_token_regs<kWide>(sm.lay, U, UH, f, a.n_words);
      }
    };
    if (sm.lay.lodd[4] > 0)
      drain(std::true_type{});
    else
      drain(std::false_type{});
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == kKMmaWarp) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ head-group streams
// A head-group stream (Sec. 5 Step 1: the g_h kv-heads of a group share one transform) projects
// the concatenated kv-heads of a group, n = 128 g_h input dims, onto n channels, held as g_h
// slice streams (slice s = storage channels s, s + g_h, ...; slice-major operand rows).  One
// persistent CTA per (group, kind, slice of 128-token items); all n channels of an item sit in
// TMEM at once (n <= 512 columns), so alpha, the maximum over all of them, is known before any
// slice is quantized.  Warp roles:
//   warp 8    : TMA producer -- per 64-dim block of the input: the 128 x 64 x tile of the group's
//               kv-heads and the n x 64 operand tile, into a 2-stage SW128 ring,
//   warp 9    : MMA issuer   -- tcgen05.mma M=128 tokens, N=256, K=16, n / 256 per k-step, into
//               the n-column accumulator,
//   warps 0-7 : two epilogue warpgroups, thread = token; warpgroup e owns slices e g_h / 2 ..:
//               their maxima meet through shared memory (an mbarrier round), then each slice is
//               quantized, the accumulator released, and the slice records packed
//               (register-resident, as aatc_encode_kernel, widths up to 8).
constexpr int kGStages = 2;
constexpr int kGXBytes = TILE * 64 * 2;            // 16 KB: 128 tokens x 64 dims
constexpr int kGEpiThreads = 256;
constexpr int kGProducerWarp = kGEpiThreads / 32;
constexpr int kGMmaWarp = kGProducerWarp + 1;
constexpr int kGThreads = kGEpiThreads + 64;

struct GroupEncodeArgs {
  const ChanEnc* enc;
  const float* inv_s;
  const StreamLayout* lay;
  int* err;
  uint32_t* words;
  float* alpha;
  int layer, n_kv, gh, n_groups, batch, start, n_tokens, n_chunks, n_words, n_tiles, ctas_per_basis;
};

template <int GH>
struct GroupEncodeSmem {
  static constexpr int N = D * GH;
  alignas(1024) unsigned char x_tile[kGStages][kGXBytes];
  alignas(1024) unsigned char u_tile[kGStages][N * 64 * 2];
  alignas(16) float inv_s[GH][D];
  alignas(16) float inv_f[GH][D];
  alignas(16) float hi[GH][D];
  alignas(16) float magic[GH][D];
  StreamLayout lay[GH];
  float xch[2][TILE];                              // per-warpgroup maxima of each token
  uint64_t full[kGStages], empty[kGStages], tfull, tempty, xbar;
  uint32_t tmem_base;
  int abort_flag;
};

template <int GH>
__global__ void __launch_bounds__(kGThreads, 1)
    aatc_encode_group_kernel(const __grid_constant__ CUtensorMap tmap_k, const __grid_constant__ CUtensorMap tmap_v,
                             const __grid_constant__ CUtensorMap tmap_g, const GroupEncodeArgs a) {
  constexpr int N = D * GH, NKB = N / 64, NH = N / 256, SPW = GH / 2;
  constexpr uint32_t kUBytes = N * 64 * 2;
  constexpr uint32_t kCols = N <= 256 ? 256 : 512;
  extern __shared__ unsigned char smem_raw[];
  auto& sm = *reinterpret_cast<GroupEncodeSmem<GH>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int basis = blockIdx.x / a.ctas_per_basis;           // (group, kind) of the layer
  const int sub = blockIdx.x % a.ctas_per_basis;
  const int grp = basis >> 1, kind = basis & 1;
  const long n_items = static_cast<long>(a.batch) * a.n_chunks;
  const long it0 = n_items * sub / a.ctas_per_basis;
  const int my_items = static_cast<int>(n_items * (sub + 1) / a.ctas_per_basis - it0);
  const CUtensorMap* tmap_x = kind == 0 ? &tmap_k : &tmap_v;
  const int row0 = ((a.layer * a.n_groups + grp) * 2 + kind) * N;   // operand rows of this stream

  for (int i = tid; i < GH * D; i += kGThreads) {
    const int sl = i / D, c = i % D;
    const int slot = (a.layer * a.n_kv + grp * GH + sl) * 2 + kind;
    const ChanEnc e = a.enc[slot * D + c];
    sm.inv_s[sl][c] = a.inv_s[slot * D + c];
    sm.inv_f[sl][c] = e.inv_f;
    sm.hi[sl][c] = e.hi;
    sm.magic[sl][c] = e.magic;
  }
  if (tid < GH) sm.lay[tid] = a.lay[(a.layer * a.n_kv + grp * GH + tid) * 2 + kind];
  if (tid == 0) {
    for (int st = 0; st < kGStages; ++st) {
      ptx::mbar_init(&sm.full[st], 1);
      ptx::mbar_init(&sm.empty[st], 1);
    }
    ptx::mbar_init(&sm.tfull, 1);
    ptx::mbar_init(&sm.tempty, kGEpiThreads);
    ptx::mbar_init(&sm.xbar, kGEpiThreads);
    sm.abort_flag = 0;
    ptx::fence_mbar_init();
  }
  if (warp == kGMmaWarp) {
    ptx::tmem_alloc(&sm.tmem_base, kCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == kGProducerWarp) {
    if (lane == 0 && my_items > 0) {
      ptx::prefetch_tmap(tmap_x);
      ptx::prefetch_tmap(&tmap_g);
      bool ok = true;
      for (int it = 0; ok && it < my_items; ++it) {
        const long item = it0 + it;
        const int b = static_cast<int>(item / a.n_chunks);
        const int t0 = static_cast<int>(item % a.n_chunks) * TILE;
        for (int kb = 0; kb < NKB; ++kb) {
          const int u = it * NKB + kb, st = u % kGStages;
          if (!ptx::mbar_wait_bounded(&sm.empty[st], ((u / kGStages) & 1) ^ 1, abort_flag)) {
            raise_abort(sm, a.err);
            ok = false;
            break;
          }
          ptx::mbar_arrive_expect_tx(&sm.full[st], kGXBytes + kUBytes);
          // the group's kv-heads are adjacent: dims grp N + 64 kb .. of the [n_kv 128]-wide rows
          ptx::tma_load_3d(sm.x_tile[st], tmap_x, &sm.full[st], grp * N + kb * 64, t0, b);
#pragma unroll
          for (int h = 0; h < NH; ++h)
            ptx::tma_load_2d(sm.u_tile[st] + h * (256 * 128), &tmap_g, &sm.full[st], kb * 64, row0 + h * 256);
        }
      }
    }
  } else if (warp == kGMmaWarp) {
    if (lane == 0 && my_items > 0) {
      constexpr uint32_t idesc = ptx::idesc_bf16_f32(128, 256);
      bool ok = true;
      for (int it = 0; ok && it < my_items; ++it) {
        if (!ptx::mbar_wait_bounded(&sm.tempty, (it & 1) ^ 1, abort_flag)) { raise_abort(sm, a.err); break; }
        ptx::tc_fence_after();
        for (int kb = 0; kb < NKB; ++kb) {
          const int u = it * NKB + kb, st = u % kGStages;
          if (!ptx::mbar_wait_bounded(&sm.full[st], (u / kGStages) & 1, abort_flag)) {
            raise_abort(sm, a.err);
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t x_base = ptx::smem_u32(sm.x_tile[st]), u_base = ptx::smem_u32(sm.u_tile[st]);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
#pragma unroll
            for (int h = 0; h < NH; ++h)
              ptx::umma_bf16(tmem + h * 256, ptx::sdesc_kmajor_sw128(x_base + kk * 32),
                             ptx::sdesc_kmajor_sw128(u_base + h * (256 * 128) + kk * 32), idesc,
                             (kb > 0 || kk > 0) ? 1u : 0u);
          ptx::umma_commit(&sm.empty[st]);
        }
        if (ok) ptx::umma_commit(&sm.tfull);
      }
    }
  } else {
    const int eg = warp >> 2, quad = warp & 3, tl = quad * 32 + lane;
    const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    uint32_t uh[8];
#pragma unroll 1
    for (int it = 0; it < my_items; ++it) {
      if (!ptx::mbar_wait_bounded(&sm.tfull, it & 1, abort_flag)) { raise_abort(sm, a.err); break; }
      ptx::tc_fence_after();
      float pm = 0.0f;
#pragma unroll
      for (int k = 0; k < SPW; ++k) {
        const int sl = eg * SPW + k;
        pm = fmaxf(pm, token_amax_regs(lane_base + sl * D, sm.inv_s[sl]));
      }
      sm.xch[eg][tl] = pm;
      ptx::mbar_arrive(&sm.xbar);                              // (a bounded wait, unlike a named barrier)
      if (!ptx::mbar_wait_bounded(&sm.xbar, it & 1, abort_flag)) { raise_abort(sm, a.err); break; }
      const float amax = fmaxf(sm.xch[0][tl], sm.xch[1][tl]);
      const float ia = amax > 0.0f ? 1.0f / amax : 0.0f;
      uint32_t U[SPW][32];
#pragma unroll
      for (int k = 0; k < SPW; ++k) {
        const int sl = eg * SPW + k;
        token_quant_regs(lane_base + sl * D, QuantTables{sm.inv_s[sl], sm.inv_f[sl], sm.hi[sl], sm.magic[sl]}, ia,
                         U[k]);
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(&sm.tempty);

      const long item = it0 + it;
      const int b = static_cast<int>(item / a.n_chunks);
      const int i = static_cast<int>(item % a.n_chunks) * TILE + tl;
      const bool ok = i < a.n_tokens;
      if (!__any_sync(0xffffffffu, ok)) continue;
      const int pos_t = a.start + i;
      if (ok && !isfinite(amax)) atomicOr(a.err, 1);
#pragma unroll
      for (int k = 0; k < SPW; ++k) {
        const int sl = eg * SPW + k;
        const size_t sidx = (static_cast<size_t>(b) * a.n_kv + grp * GH + sl) * 2 + kind;
        if (ok) a.alpha[sidx * a.n_tiles * TILE + pos_t] = amax;
        RecordFlush f{a.words + sidx * stream_words + static_cast<size_t>(pos_t / TILE) * a.n_words * TILE,
                      pos_t % TILE, kind == 1, ok, 0};
        pack_token_regs<false>(sm.lay[sl], U[k], uh, f, a.n_words);
      }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == kGMmaWarp) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kCols);
  }
}

// ------------------------------------------------------------------ encode from hidden states
// Sec. 5 Step 1 caches H = X A, the coefficients computed from the layer input x rather than
// from k = x W.  With A_hat = W U (the plan basis, = A sqrt(S) up to channel order) the MMA
// gives h = x A_hat = k U directly, K = d_model.  One persistent CTA per (kv-head, slice of
// 128-token tiles); warp roles as aatc_encode_kernel:
//   warp 16   : TMA producer -- per 64-wide d_model block: the 128 x 64 x tile and the 256 x 64
//               A_hat tile of the head's key and value channels (two 128-row boxes, one operand),
//   warp 17   : MMA issuer   -- tcgen05.mma M=128 tokens, N=256 (key | value channels), K=16,
//               into one of two 256-column TMEM accumulators,
//   warps 0-15: four epilogue groups (stream = group & 1, accumulator = group >> 1), thread =
//               token: the quantize / pack epilogue of aatc_encode_kernel.
// CTA i takes kv-head i mod H and tiles i / H, i / H + J, ... (J CTAs per head), so the H CTAs
// working on one token tile at a time read its x block from L2 after the first.
constexpr int kHStages = 3;
constexpr int kHK = 64;                            // d_model elements per stage (one 128-byte row)
constexpr int kHXBytes = TILE * kHK * 2;           // 16 KB
constexpr int kHABytes = 2 * D * kHK * 2;          // 32 KB

struct EncodeHiddenArgs {
  const ChanEnc* enc;
  const float* inv_s;
  const StreamLayout* lay;
  int* err;
  uint32_t* words;
  float* alpha;
  int layer, n_kv, batch, start, n_tokens, n_chunks, n_words, n_tiles, d_model;
};

struct EncodeHiddenSmem {
  alignas(1024) unsigned char x_tile[kHStages][kHXBytes];
  alignas(1024) unsigned char a_tile[kHStages][kHABytes];
  ChanEnc enc[2][D];
  float inv_s[2][D];
  StreamLayout lay[2];
  uint32_t ubytes[kEpiThreads][kByteRow / 4];
  uint64_t full[kHStages], empty[kHStages], tfull[2], tempty[2];
  uint32_t tmem_base;
  int abort_flag;
};

__global__ void __launch_bounds__(kThreads, 1)
    aatc_encode_hidden_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_a,
                              const EncodeHiddenArgs a) {
  extern __shared__ unsigned char smem_raw[];
  EncodeHiddenSmem& sm =
      *reinterpret_cast<EncodeHiddenSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int head = blockIdx.x % a.n_kv, j = blockIdx.x / a.n_kv, J = gridDim.x / a.n_kv;
  const long n_items = static_cast<long>(a.batch) * a.n_chunks;
  const int my_items = n_items > j ? static_cast<int>((n_items - 1 - j) / J + 1) : 0;
  const int nk = a.d_model / kHK;
  const int sk = (a.layer * a.n_kv + head) * 2;                // key stream; values sk + 1

  for (int i = tid; i < 2 * D; i += kThreads) {
    sm.enc[i >> 7][i & (D - 1)] = a.enc[sk * D + i];
    sm.inv_s[i >> 7][i & (D - 1)] = a.inv_s[sk * D + i];
  }
  if (tid == 0) {
    sm.lay[0] = a.lay[sk];
    sm.lay[1] = a.lay[sk + 1];
    for (int s = 0; s < kHStages; ++s) {
      ptx::mbar_init(&sm.full[s], 1);
      ptx::mbar_init(&sm.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(&sm.tfull[b], 1);
      ptx::mbar_init(&sm.tempty[b], 256);
    }
    sm.abort_flag = 0;
    ptx::fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    ptx::tmem_alloc(&sm.tmem_base, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == kProducerWarp) {
    if (lane == 0 && my_items > 0) {
      ptx::prefetch_tmap(&tmap_x);
      ptx::prefetch_tmap(&tmap_a);
      bool ok = true;
      for (int it = 0; ok && it < my_items; ++it) {
        const long tile = j + static_cast<long>(it) * J;
        const int b = static_cast<int>(tile / a.n_chunks);
        const int t0 = static_cast<int>(tile % a.n_chunks) * TILE;
        for (int ks = 0; ks < nk; ++ks) {
          const int u = it * nk + ks, s = u % kHStages;
          const uint32_t ph = (u / kHStages) & 1;
          if (!ptx::mbar_wait_bounded(&sm.empty[s], ph ^ 1, abort_flag)) { raise_abort(sm, a.err); ok = false; break; }
          ptx::mbar_arrive_expect_tx(&sm.full[s], kHXBytes + kHABytes);
          ptx::tma_load_3d(sm.x_tile[s], &tmap_x, &sm.full[s], ks * kHK, t0, b);
          ptx::tma_load_2d(sm.a_tile[s], &tmap_a, &sm.full[s], ks * kHK, sk * D);
          ptx::tma_load_2d(sm.a_tile[s] + kHABytes / 2, &tmap_a, &sm.full[s], ks * kHK, (sk + 1) * D);
        }
      }
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0 && my_items > 0) {
      constexpr uint32_t idesc = ptx::idesc_bf16_f32(128, 2 * D);
      bool ok = true;
      for (int it = 0; ok && it < my_items; ++it) {
        const int bf = it & 1;
        if (!ptx::mbar_wait_bounded(&sm.tempty[bf], ((it >> 1) & 1) ^ 1, abort_flag)) { raise_abort(sm, a.err); break; }
        ptx::tc_fence_after();
        for (int ks = 0; ks < nk; ++ks) {
          const int u = it * nk + ks, s = u % kHStages;
          const uint32_t ph = (u / kHStages) & 1;
          if (!ptx::mbar_wait_bounded(&sm.full[s], ph, abort_flag)) { raise_abort(sm, a.err); ok = false; break; }
          ptx::tc_fence_after();
          const uint32_t x_base = ptx::smem_u32(sm.x_tile[s]), a_base = ptx::smem_u32(sm.a_tile[s]);
#pragma unroll
          for (int kk = 0; kk < kHK / 16; ++kk)
            ptx::umma_bf16(tmem + 2 * D * bf, ptx::sdesc_kmajor_sw128(x_base + kk * 32),
                           ptx::sdesc_kmajor_sw128(a_base + kk * 32), idesc, (ks > 0 || kk > 0) ? 1u : 0u);
          ptx::umma_commit(&sm.empty[s]);
        }
        if (ok) ptx::umma_commit(&sm.tfull[bf]);
      }
    }
  } else {
    const int eg = warp >> 2, sidx = eg & 1, bf = eg >> 1;
    const int quad = warp & 3;
    const int tl = quad * 32 + lane;
    const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;
    const StreamLayout& lay = sm.lay[sidx];
    uint32_t* my_bytes = sm.ubytes[tid];
    for (int it = bf; it < my_items; it += 2) {
      if (!ptx::mbar_wait_bounded(&sm.tfull[bf], (it >> 1) & 1, abort_flag)) { raise_abort(sm, a.err); break; }
      ptx::tc_fence_after();
      const uint32_t taddr = tmem + 2 * D * bf + D * sidx + (static_cast<uint32_t>(quad * 32) << 16);
      const float amax = quantize_token(taddr, sm.enc[sidx], sm.inv_s[sidx], my_bytes);
      ptx::tc_fence_before();
      ptx::mbar_arrive(&sm.tempty[bf]);

      const long tile = j + static_cast<long>(it) * J;
      const int b = static_cast<int>(tile / a.n_chunks);
      const int i = static_cast<int>(tile % a.n_chunks) * TILE + tl;     // input token index
      if (i >= a.n_tokens) continue;
      const int pos_t = a.start + i;
      const size_t cs = (static_cast<size_t>(b) * a.n_kv + head) * 2 + sidx;
      if (!isfinite(amax)) atomicOr(a.err, 1);
      a.alpha[cs * a.n_tiles * TILE + pos_t] = amax;
      pack_token(lay, my_bytes, record_writer(a.words, cs, stream_words, a.n_words, pos_t, sidx == 1), a.n_words);
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// K or V: bf16 [batch][n_tokens][n_kv][128]; box = 64 dims x 1 head x 128 tokens x 1 sequence.
cudaError_t make_kv_map(CUtensorMap* map, const void* base, int batch, int n_tokens, int n_kv) {
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(n_kv),
                              static_cast<cuuint64_t>(n_tokens), static_cast<cuuint64_t>(batch)};
  const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(n_kv) * D * 2,
                                 static_cast<cuuint64_t>(n_tokens) * n_kv * D * 2};
  const cuuint32_t box[4] = {64, 1, TILE, 1};
  const cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

cudaError_t make_tensor_map_2d(void* map, bool f16, const void* base, uint64_t inner, uint64_t rows,
                               uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_bytes)};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t es[2] = {1, 1};
  CUresult r = enc(reinterpret_cast<CUtensorMap*>(map),
                   f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                   const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t encode_tensor_maps_u(Plan& plan) {
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  auto* map = reinterpret_cast<CUtensorMap*>(plan.tmap_u);
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(plan.n_streams) * D};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(D) * 2};
  const cuuint32_t box[2] = {64, TILE};
  const cuuint32_t es[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(plan.dev.ubf16_t), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  plan.tmap_ok = r == CUDA_SUCCESS;
  return plan.tmap_ok ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t launch_encode(const Plan& plan, int layer, const void* K, const void* V, int batch, int start,
                          int n_tokens, void* cache, int max_tokens, cudaStream_t st) {
  static_assert(sizeof(CUtensorMap) == 128, "CUtensorMap size");
  CUtensorMap mk, mv;
  cudaError_t e = make_kv_map(&mk, K, batch, n_tokens, plan.dims.n_kv_heads);
  if (e == cudaSuccess) e = make_kv_map(&mv, V, batch, n_tokens, plan.dims.n_kv_heads);
  if (e != cudaSuccess) return e;
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  EncodeArgs a;
  a.enc = plan.dev.enc;
  a.inv_s = plan.dev.inv_s;
  a.lay = plan.dev.lay;
  a.entry = plan.dev.entry;
  a.err = plan.dev.err;
  a.n_entries = plan.n_entries;
  a.words = static_cast<uint32_t*>(cache);
  a.alpha = reinterpret_cast<float*>(static_cast<uint32_t*>(cache) + g.words_elems);
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.batch = batch;
  a.start = start;
  a.n_tokens = n_tokens;
  a.n_chunks = (n_tokens + TILE - 1) / TILE;
  a.n_words = plan.n_words;
  a.n_tiles = g.n_tiles;
  const int n_basis = 2 * plan.dims.n_kv_heads;
  const long items_per_basis = static_cast<long>(batch) * a.n_chunks;
  int k = std::max(1, plan.num_sms / n_basis);
  if (k > items_per_basis) k = static_cast<int>(items_per_basis);
  a.ctas_per_basis = k;
  const size_t smem = sizeof(EncodeSmem) + 1024;
  e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_encode_kernel), smem);
  if (e != cudaSuccess) return e;
  const auto* mu = reinterpret_cast<const CUtensorMap*>(plan.tmap_u);
  aatc_encode_kernel<<<n_basis * k, kKThreads, smem, st>>>(mk, mv, *mu, a);
  return cudaGetLastError();
}


cudaError_t launch_encode_hidden(const Plan& plan, int layer, const void* x, int d_model, const void* a_hat,
                                 int batch, int start, int n_tokens, void* cache, int max_tokens, cudaStream_t st) {
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap mx, ma;
  {
    // x: bf16 [batch][n_tokens][d_model]; box 64 x 128 tokens x 1 (rows past n_tokens read 0)
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(d_model), static_cast<cuuint64_t>(n_tokens),
                                static_cast<cuuint64_t>(batch)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(d_model) * 2,
                                   static_cast<cuuint64_t>(n_tokens) * d_model * 2};
    const cuuint32_t box[3] = {kHK, TILE, 1};
    const cuuint32_t es[3] = {1, 1, 1};
    if (enc(&mx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(x), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    // A_hat: bf16 [L * H * 2 * 128 rows][d_model]; box 64 x 128 rows
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(d_model), static_cast<cuuint64_t>(plan.n_streams) * D};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(d_model) * 2};
    const cuuint32_t box[2] = {kHK, TILE};
    const cuuint32_t es[2] = {1, 1};
    if (enc(&ma, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a_hat), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  EncodeHiddenArgs a;
  a.enc = plan.dev.enc;
  a.inv_s = plan.dev.inv_s;
  a.lay = plan.dev.lay;
  a.err = plan.dev.err;
  a.words = static_cast<uint32_t*>(cache);
  a.alpha = reinterpret_cast<float*>(static_cast<uint32_t*>(cache) + g.words_elems);
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.batch = batch;
  a.start = start;
  a.n_tokens = n_tokens;
  a.n_chunks = (n_tokens + TILE - 1) / TILE;
  a.n_words = plan.n_words;
  a.n_tiles = g.n_tiles;
  a.d_model = d_model;
  const long n_items = static_cast<long>(batch) * a.n_chunks;
  long per_head = std::max(1, plan.num_sms / a.n_kv);
  per_head = std::min(per_head, n_items);
  const size_t smem = sizeof(EncodeHiddenSmem) + 1024;
  cudaError_t e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_encode_hidden_kernel), smem);
  if (e != cudaSuccess) return e;
  aatc_encode_hidden_kernel<<<static_cast<unsigned>(per_head * a.n_kv), kThreads, smem, st>>>(mx, ma, a);
  return cudaGetLastError();
}

cudaError_t launch_group_encode(const Plan& plan, int layer, const void* K, const void* V, int batch, int start,
                                int n_tokens, void* cache, int max_tokens, cudaStream_t st) {
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  const int gh = plan.group_heads, n_kv = plan.dims.n_kv_heads;
  if (gh != 2 && gh != 4) return cudaErrorNotSupported;
  CUtensorMap mk, mv;
  // K or V as bf16 [batch][n_tokens][n_kv * 128]: box 64 dims x 128 tokens x 1 sequence
  for (int kind = 0; kind < 2; ++kind) {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(n_kv) * D, static_cast<cuuint64_t>(n_tokens),
                                static_cast<cuuint64_t>(batch)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(n_kv) * D * 2,
                                   static_cast<cuuint64_t>(n_tokens) * n_kv * D * 2};
    const cuuint32_t box[3] = {64, TILE, 1};
    const cuuint32_t es[3] = {1, 1, 1};
    if (enc(kind == 0 ? &mk : &mv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(kind == 0 ? K : V), dims,
            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const CacheGeom g = cache_geom(batch, n_kv, max_tokens, plan.n_words);
  GroupEncodeArgs a;
  a.enc = plan.dev.enc;
  a.inv_s = plan.dev.inv_s;
  a.lay = plan.dev.lay;
  a.err = plan.dev.err;
  a.words = static_cast<uint32_t*>(cache);
  a.alpha = reinterpret_cast<float*>(static_cast<uint32_t*>(cache) + g.words_elems);
  a.layer = layer;
  a.n_kv = n_kv;
  a.gh = gh;
  a.n_groups = n_kv / gh;
  a.batch = batch;
  a.start = start;
  a.n_tokens = n_tokens;
  a.n_chunks = (n_tokens + TILE - 1) / TILE;
  a.n_words = plan.n_words;
  a.n_tiles = g.n_tiles;
  const int n_basis = 2 * a.n_groups;
  const long items = static_cast<long>(batch) * a.n_chunks;
  long k = std::max(1, plan.num_sms / n_basis);
  a.ctas_per_basis = static_cast<int>(std::min(k, items));
  const auto* mg = reinterpret_cast<const CUtensorMap*>(plan.tmap_g);
  const unsigned grid = static_cast<unsigned>(n_basis * a.ctas_per_basis);
  if (gh == 2) {
    const size_t smem = sizeof(GroupEncodeSmem<2>) + 1024;
    cudaError_t e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_encode_group_kernel<2>), smem);
    if (e != cudaSuccess) return e;
    aatc_encode_group_kernel<2><<<grid, kGThreads, smem, st>>>(mk, mv, *mg, a);
  } else {
    const size_t smem = sizeof(GroupEncodeSmem<4>) + 1024;
    cudaError_t e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_encode_group_kernel<4>), smem);
    if (e != cudaSuccess) return e;
    aatc_encode_group_kernel<4><<<grid, kGThreads, smem, st>>>(mk, mv, *mg, a);
  }
  return cudaGetLastError();
}

}  // namespace aatc
