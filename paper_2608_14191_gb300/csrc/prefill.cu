// Prefill attention over the packed cache: a chunk of new query tokens attends causally to the
// cached tokens (Def. sdpa for every query row; Algorithm 1's reconstruct / attend lines, computed
// in the transformed space as the decode does: q . (U h) = (U^T q) . h).
//
// Two launches per call:
//   codes    per (128-token tile, kv-head x K|V, sequence): the packed records -> the signed codes
//            code_c = u_c - 2^(b_c - 1) as f16 (exact: |code| <= 128) in a workspace of rows of 128
//            f16, [b][h][K|V][n_ctx_pad][128]: key rows are tokens, value tiles are stored
//            transposed ([tile][channel][token]) so both are K-major tensor-core operands;
//   attn     per (128 query rows, kv-head, sequence), rows = (query token, head of the GQA group),
//            everything on the tensor cores (tcgen05): q' = (U_K^T q) f^K log2(e) / sqrt(128),
//            per 128-token tile S = alpha^K (q'_hi + q'_lo) . code^K, causal mask, lazily
//            rescaled softmax, P' = 2^(S - m) alpha^V (f16) and O += P' code^V, finally
//            out = U_V (f^V O / l).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "aatc_internal.h"
#include "ptx.cuh"

namespace aatc {
namespace {

constexpr float kPLog2e = 1.4426950408889634f;
constexpr float kPOpMax = 16384.0f; // q' rows scaled so the largest |value| is 2^14

struct PrefillArgs {
  const uint32_t* words;     // cache word region (this layer)
  const float* alpha;        // cache alpha region
  const __nv_bfloat16* q;    // [batch][n_q][H_q][128]
  float* out;                // [batch][n_q][H_q][128]
  __half* codes;             // workspace [batch][n_kv][2][n_ctx_pad][128]
  const float* u32;          // plan: [S][128 dim][128 ch]
  const float* u32t;         // plan: [S][128 ch][128 dim]
  const float* f;            // plan: [S][128]
  const ChanEnc* enc;        // plan: [S][128] (offsets 2^(b-1))
  const StreamLayout* lay;   // plan: [S]
  const short* entry;        // plan: [S][n_entries]
  const short* chan_ent;     // plan: [S][128][kChanEnt]
  int layer, n_kv, n_q_heads, group, q_start, n_q, n_ctx, n_ctx_pad, n_tiles, n_words, n_entries;
  int* err;
};

__global__ void __launch_bounds__(TILE) aatc_prefill_codes_kernel(const PrefillArgs a) {
  __shared__ uint32_t rec[32][TILE];           // record words of the tile's tokens (W <= 32)
  const int tile = blockIdx.x, hk = blockIdx.y, b = blockIdx.z, t = threadIdx.x;
  const int head = hk >> 1, kind = hk & 1;
  const size_t cs = (static_cast<size_t>(b) * a.n_kv + head) * 2 + kind;
  const int tok = tile * TILE + t;
  __half* dst = a.codes + (cs * a.n_ctx_pad + tok) * D;
  if (tok >= a.n_ctx) {                        // padding rows of the last tile: zero codes
    if (tok < a.n_ctx_pad) {
      if (kind == 1) {
        __half* d2 = a.codes + cs * a.n_ctx_pad * D + static_cast<size_t>(tile) * TILE * D + t;
        for (int c = 0; c < D; ++c) d2[c * TILE] = __float2half_rn(0.0f);
      } else {
        for (int c = 0; c < D; c += 8) *reinterpret_cast<uint4*>(dst + c) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    return;
  }
  const int s = (a.layer * a.n_kv + head) * 2 + kind;
  const StreamLayout ly = a.lay[s];
  const int nw = ly.n2 / 16 + (ly.n1 + 31) / 32;
  const uint32_t* tw = a.words + (cs * a.n_tiles + tile) * static_cast<size_t>(a.n_words) * TILE;
  for (int w = 0; w < nw; ++w) {
    const uint32_t* ww = tw + static_cast<size_t>(w) * TILE;
    uint32_t x;
    if (kind == 0) {
      x = ww[t];
    } else {                                   // quad-interleaved: quarter r in slot 4Q + (0, 2, 1, 3)[r]
      const int q4 = 4 * (t >> 2), sh = 8 * (t & 3);
      x = ((ww[q4] >> sh) & 0xFFu) | (((ww[q4 + 2] >> sh) & 0xFFu) << 8) | (((ww[q4 + 1] >> sh) & 0xFFu) << 16) |
          (((ww[q4 + 3] >> sh) & 0xFFu) << 24);
    }
    rec[w][t] = x;                             // each thread reads back only its own column
  }
  const short* ce = a.chan_ent + static_cast<size_t>(s) * D * kChanEnt;
  const short* ent = a.entry + static_cast<size_t>(s) * a.n_entries;
  // values for the tensor-core kernel: per 128-token tile [channel][token]
  __half* dst_t = a.codes + cs * a.n_ctx_pad * D + static_cast<size_t>(tile) * TILE * D + t;
  const bool transposed = kind == 1;
  for (int c = 0; c < D; c += 2) {
    float v2[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int cc = c + i;
      uint32_t u = 0;
      for (int k = 0; k < kChanEnt; ++k) {
        const int e = ce[cc * kChanEnt + k];
        if (e < 0) break;
        uint32_t v;
        if (e < ly.n2) {
          v = (rec[e >> 4][t] >> (2 * (e & 15))) & 3u;
        } else {
          const int e1 = e - ly.n2;
          v = (rec[ly.n2 / 16 + (e1 >> 5)][t] >> (e1 & 31)) & 1u;
        }
        u |= v << ((ent[e] >> 8) & 15);
      }
      v2[i] = static_cast<float>(u) - a.enc[s * D + cc].off;   // dropped channels: u = off = 0
    }
    if (transposed) {
      dst_t[c * TILE] = __float2half_rn(v2[0]);
      dst_t[(c + 1) * TILE] = __float2half_rn(v2[1]);
    } else {
      *reinterpret_cast<__half2*>(dst + c) = __floats2half2_rn(v2[0], v2[1]);
    }
  }
}

__device__ __forceinline__ float ex2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// ---------------------------------------------------------------- tensor-core (tcgen05) attention
// Per CTA 128 query rows (= TMEM lanes) of one (kv-head, sequence).  Warps 0-7 do the softmax:
// warp w owns TMEM lanes 32 (w & 3) .. + 31 and the column half w >> 2 of every 128-column TMEM
// block.  Warp 8 is the control warp: one thread issues every TMA copy and tensor-core MMA and
// talks to the softmax warps through mbarriers only.
//   prologue  q' = (q U_K) f^K log2(e) / sqrt(128) on the tensor cores: q (bf16, exact) against
//             U_K split into three bf16 parts (about 2^-25 relative), rows scaled to 2^14 and
//             split into f16 hi / lo operands kept in TMEM (the A operand of the score MMA, so
//             only the key tile is read from shared memory)
//   per 128-token tile (TMA, 128-byte swizzle, key and value tiles double-buffered):
//             S = q'_hi . code_K + q'_lo . code_K   tcgen05.mma M = N = 128, K = 128; the softmax
//             keeps its scores in registers, so S of tile t + 1 is computed into the same TMEM
//             columns as soon as every warp has read S(t)
//             softmax from TMEM with the scores held in registers between the maximum and the
//             exponent: s = S rs alpha^K (causal mask), lazy maximum (O rescaled only when a
//             row's maximum grows by more than 2^8, so P' = 2^(s - m) alpha^V stays inside f16)
//             P' stored to TMEM as f16 pairs: the A operand of O += P' . code_V^T
//   epilogue  out = (f^V O / l) U_V^T on the tensor cores, both operands split hi / lo in bf16.
constexpr int kTRows = 128;
constexpr int kTSoftmax = 256;                     // softmax threads (warps 0-7)
constexpr int kTThreads = kTSoftmax + 32;          // + the control warp
constexpr int kTCtl = kTSoftmax;                   // the thread that issues copies and MMAs
constexpr int kTAtom = 128 * 128;                  // one 128-row K-atom (64 16-bit values per row)
constexpr int kTOp = 2 * kTAtom;                   // one 128 x 128 16-bit operand (two K-atoms)
constexpr float kLazyLog2 = 8.0f;
constexpr uint32_t kIdescTT = ptx::idesc_f16_f32(128, 128);
constexpr uint32_t kIdescBB = ptx::idesc_bf16_f32(128, 128);
constexpr uint32_t kColS = 0;                      // score buffer; projection results
constexpr uint32_t kColO = 128;                    // O accumulator
constexpr uint32_t kColP = 256;                    // two P' buffers (256, 320): 64 columns of f16 pairs
constexpr uint32_t kColQ = 384;                    // q' hi (384) and lo (448): A operands of the score MMA

struct PrefillTcSmem {
  alignas(1024) unsigned char kt[2][kTOp];         // key codes: K-atoms = channels, rows = tokens
  alignas(1024) unsigned char vt[2][kTOp];         // value codes: K-atoms = tokens 0-63 | 64-127, rows = channels
  float al[3][2][TILE];                            // alpha^K, alpha^V of three tiles
  float xch[2][2][kTRows];                         // per-row partials of the two column halves (two slots)
  uint64_t bar_k[2], bar_v[2], ofree[2], bar_s, sfree, pready, bar_p;
  uint32_t tmem;
  int abort_flag;
};
// kt and vt together hold the four projection operands (prologue, epilogue)
static_assert(offsetof(PrefillTcSmem, vt) == offsetof(PrefillTcSmem, kt) + 2 * kTOp, "operand slots contiguous");

// byte offset of element (row, k) of a 128-row K-major operand with the 128-byte swizzle
__device__ __forceinline__ int sw128_off(int row, int k) {
  return (k >> 6) * kTAtom + (row >> 3) * 1024 + (row & 7) * 128 + ((((k & 63) >> 3) ^ (row & 7)) << 4) + (k & 7) * 2;
}

__device__ __forceinline__ uint32_t pack_bf2(__nv_bfloat16 lo, __nv_bfloat16 hi) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(lo)) | (static_cast<uint32_t>(__bfloat16_as_ushort(hi)) << 16);
}

// 8 fp32 values -> `parts` bf16 parts (u = p0 + p1 + p2 up to the last part's rounding), each
// stored as one 16-byte granule at dst[i * kTOp]
__device__ __forceinline__ void store_split_bf16(unsigned char* dst, const float (&u)[8], int parts) {
  uint32_t w[3][4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    float x0 = u[2 * j], x1 = u[2 * j + 1];
#pragma unroll
    for (int p = 0; p < 3; ++p) {
      const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
      w[p][j] = pack_bf2(h0, h1);
      x0 -= __bfloat162float(h0);
      x1 -= __bfloat162float(h1);
    }
  }
#pragma unroll
  for (int p = 0; p < 3; ++p)
    if (p < parts) *reinterpret_cast<uint4*>(dst + p * kTOp) = make_uint4(w[p][0], w[p][1], w[p][2], w[p][3]);
}

// barrier among the softmax warps only
__device__ __forceinline__ void softmax_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kTSoftmax) : "memory"); }

__global__ void __launch_bounds__(kTThreads, 1)
    aatc_prefill_tc_kernel(const __grid_constant__ CUtensorMap tm, const PrefillArgs a) {
  extern __shared__ unsigned char smraw[];
  PrefillTcSmem& sm =
      *reinterpret_cast<PrefillTcSmem*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  // row blocks in reverse: the longest causal ranges start first, the shortest fill the tail
  const int rb = gridDim.x - 1 - blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool softmax = tid < kTSoftmax;
  const int G = a.group, n_rows = a.n_q * G;
  const int sk = (a.layer * a.n_kv + head) * 2, sv = sk + 1;
  const size_t csk = (static_cast<size_t>(b) * a.n_kv + head) * 2, csv = csk + 1;
  const int R0 = rb * kTRows;
  const int r_last = min(n_rows - 1, R0 + kTRows - 1) - R0;
  const int kv_end = min(a.n_ctx, a.q_start + (R0 + r_last) / G + 1);
  const int n_kv_tiles = (kv_end + TILE - 1) / TILE;
  const int r = 32 * (warp & 3) + lane, half = (warp >> 2) & 1, hc = 64 * half;
  const uint32_t lane_base = static_cast<uint32_t>(32 * (warp & 3)) << 16;
  const int R = R0 + r;
  unsigned char* const pj = sm.kt[0];              // projection operand i at pj + i * kTOp
  volatile int* abort_flag = &sm.abort_flag;
  auto wait = [&](uint64_t* bar, uint32_t parity) {
    if (!ptx::mbar_wait_bounded(bar, parity, abort_flag)) {
      sm.abort_flag = 1;
      atomicOr(a.err, 2);
    }
  };

  if (tid == kTCtl) {
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(&sm.bar_k[i], 1);
      ptx::mbar_init(&sm.bar_v[i], 1);
      ptx::mbar_init(&sm.ofree[i], 1);          // PV of tiles i, i + 2, ... done
    }
    ptx::mbar_init(&sm.bar_s, 1);                    // S(t) computed
    ptx::mbar_init(&sm.sfree, kTSoftmax / 32);       // S(t) read out by every softmax warp
    ptx::mbar_init(&sm.pready, kTSoftmax / 32);
    ptx::mbar_init(&sm.bar_p, 1);
    sm.abort_flag = 0;
    ptx::fence_mbar_init();
    ptx::prefetch_tmap(&tm);
  }
  if (warp == 0) {
    ptx::tmem_alloc(&sm.tmem, 512);
    ptx::tmem_relinquish();
  }
  // ---- projection operands: q rows (bf16) in slot 0, U_K^T (rows = channel, K = dim) in three
  // bf16 parts in slots 1-3
  if (softmax) {
    for (int g = tid; g < kTRows * 16; g += kTSoftmax) {
      const int row = g >> 4, k8 = (g & 15) * 8, RR = R0 + row;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (RR < n_rows) {
        const int qi = RR / G, qh = head * G + RR % G;
        v = *reinterpret_cast<const uint4*>(a.q + ((static_cast<size_t>(b) * a.n_q + qi) * a.n_q_heads + qh) * D +
                                            k8);
      }
      *reinterpret_cast<uint4*>(pj + sw128_off(row, k8)) = v;
    }
    const float* ukt = a.u32t + static_cast<size_t>(sk) * D * D;
    for (int g = tid; g < D * 16; g += kTSoftmax) {
      const int c = g >> 4, k8 = (g & 15) * 8;
      const float4 u0 = *reinterpret_cast<const float4*>(ukt + c * D + k8);
      const float4 u1 = *reinterpret_cast<const float4*>(ukt + c * D + k8 + 4);
      const float u[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
      store_split_bf16(pj + kTOp + sw128_off(c, k8), u, 3);
    }
  }
  ptx::fence_proxy_async_smem();
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sm.tmem;
  const uint32_t pj_a = ptx::smem_u32(pj);
  if (tid == kTCtl) {
#pragma unroll 1
    for (int part = 0; part < 3; ++part)
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t off = (kk >> 2) * kTAtom + (kk & 3) * 32;
        ptx::umma_bf16(tmem + kColS, ptx::sdesc_kmajor_sw128(pj_a + off),
                       ptx::sdesc_kmajor_sw128(pj_a + (1 + part) * kTOp + off), kIdescBB, (part | kk) ? 1u : 0u);
      }
    ptx::umma_commit(&sm.bar_p);
  }
  // ---- q' rows scaled to 2^14, f16 hi / lo into the score operands
  float rsr = 1.0f;
  if (softmax) {
    wait(&sm.bar_p, 0);
    ptx::tc_fence_after();
    uint32_t q0[32], q1[32];
    ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc, q0);
    ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc + 32, q1);
    ptx::tmem_ld_wait();
    ptx::tmem_regs_ready(q0);
    ptx::tmem_regs_ready(q1);
    const float sc = kPLog2e * 0.08838834764831845f;
    const float* fk = a.f + sk * D + hc;
    float x[64];
    float m = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      x[i] = __uint_as_float(q0[i]) * fk[i] * sc;
      x[32 + i] = __uint_as_float(q1[i]) * fk[32 + i] * sc;
      m = fmaxf(m, fmaxf(fabsf(x[i]), fabsf(x[32 + i])));
    }
    sm.xch[0][half][r] = m;
    softmax_sync();
    m = fmaxf(sm.xch[0][0][r], sm.xch[0][1][r]);
    const float inv = m > 0.0f ? kPOpMax / m : 0.0f;
    rsr = m > 0.0f ? m / kPOpMax : 1.0f;             // > 0, so the mask's -inf survives the scaling
    // this thread's 64 channels as 32 f16 pairs of hi and of lo: TMEM columns kColQ + 32 half ..
    // (hi) and kColQ + 64 + 32 half .. (lo), row = lane
    uint32_t hw[32], lw[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float y0 = x[2 * j] * inv, y1 = x[2 * j + 1] * inv;
      const __half2 h = __floats2half2_rn(y0, y1);
      const float2 hf = __half22float2(h);
      hw[j] = *reinterpret_cast<const uint32_t*>(&h);
      lw[j] = pack_h2(y0 - hf.x, y1 - hf.y);
    }
    ptx::tmem_st32(tmem + lane_base + kColQ + 32 * half, hw);
    ptx::tmem_st32(tmem + lane_base + kColQ + 64 + 32 * half, lw);
    ptx::tmem_wait_st();
  }
  // alpha^K / alpha^V of one tile: thread tid < 256 owns entry tid (K for tid < 128)
  auto alpha_of = [&](int t) -> float {
    const int tl = tid & (TILE - 1), tok = t * TILE + tl;
    const size_t cs = tid < TILE ? csk : csv;
    return tok < a.n_ctx ? a.alpha[cs * a.n_tiles * TILE + tok] : 0.0f;
  };
  float a_next = 0.0f;
  if (softmax && n_kv_tiles > 0) {
    sm.al[0][tid >> 7][tid & (TILE - 1)] = alpha_of(0);
    if (n_kv_tiles > 1) a_next = alpha_of(1);
  }
  ptx::fence_proxy_async_smem();
  ptx::tc_fence_before();
  __syncthreads();                                        // q' and alpha of tile 0 complete; slots, S free
  ptx::tc_fence_after();

  if (!softmax) {
    // ---- control thread: TMA copies and MMAs.  Every wait below is on a phase that cannot be
    // overtaken: the next arrival on that barrier needs an action this thread takes later.
    if (lane == 0 && n_kv_tiles > 0) {
      auto load_k = [&](int t) {
        const int buf = t & 1;
        const int krow = static_cast<int>(csk * a.n_ctx_pad) + t * TILE;
        ptx::mbar_arrive_expect_tx(&sm.bar_k[buf], kTOp);
        ptx::tma_load_2d(sm.kt[buf], &tm, &sm.bar_k[buf], 0, krow);
        ptx::tma_load_2d(sm.kt[buf] + kTAtom, &tm, &sm.bar_k[buf], 64, krow);
      };
      auto load_v = [&](int t) {
        const int buf = t & 1;
        const int vrow = static_cast<int>(csv * a.n_ctx_pad) + t * TILE;
        ptx::mbar_arrive_expect_tx(&sm.bar_v[buf], kTOp);
        ptx::tma_load_2d(sm.vt[buf], &tm, &sm.bar_v[buf], 0, vrow);
        ptx::tma_load_2d(sm.vt[buf] + kTAtom, &tm, &sm.bar_v[buf], 64, vrow);
      };
      auto issue_s = [&](int t) {                       // S = q'_hi . code_K + q'_lo . code_K, A from TMEM
        const uint32_t kt_a = ptx::smem_u32(sm.kt[t & 1]);
        ptx::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * kTAtom + (kk & 3) * 32;
          ptx::umma_f16_ta(tmem + kColS, tmem + kColQ + 8 * kk, ptx::sdesc_kmajor_sw128(kt_a + off), kIdescTT,
                           kk > 0 ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * kTAtom + (kk & 3) * 32;
          ptx::umma_f16_ta(tmem + kColS, tmem + kColQ + 64 + 8 * kk, ptx::sdesc_kmajor_sw128(kt_a + off), kIdescTT,
                           1u);
        }
        ptx::umma_commit(&sm.bar_s);
      };
      load_k(0);
      load_v(0);
      if (n_kv_tiles > 1) {
        load_k(1);
        load_v(1);
      }
      wait(&sm.bar_k[0], 0);
      issue_s(0);
      for (int t = 0; t < n_kv_tiles; ++t) {
        const int buf = t & 1;
        if (t + 1 < n_kv_tiles) {
          wait(&sm.sfree, t & 1);                       // S(t) read out: the S buffer and kt[buf] are free
          if (t + 2 < n_kv_tiles) load_k(t + 2);
          wait(&sm.bar_k[buf ^ 1], ((t + 1) >> 1) & 1);
          issue_s(t + 1);
          if (t >= 1) {                                 // PV(t - 1) has read vt[buf ^ 1]
            wait(&sm.ofree[buf ^ 1], ((t - 1) >> 1) & 1);
            load_v(t + 1);
          }
        }
        wait(&sm.pready, t & 1);
        wait(&sm.bar_v[buf], (t >> 1) & 1);
        ptx::tc_fence_after();
        const uint32_t vt_a = ptx::smem_u32(sm.vt[buf]);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * kTAtom + (kk & 3) * 32;
          ptx::umma_f16_ta(tmem + kColO, tmem + kColP + 64 * buf + 8 * kk, ptx::sdesc_kmajor_sw128(vt_a + off),
                           kIdescTT, (t > 0 || kk > 0) ? 1u : 0u);
        }
        ptx::umma_commit(&sm.ofree[buf]);
      }
    }
    __syncwarp();                                         // the control warp reconverges
  } else {
    // ---- softmax warps
    const int pos = R < n_rows ? a.q_start + R / G : -1;   // padding rows attend to nothing
    const int last = min(pos, a.n_ctx - 1);               // last token this row attends to
    float m_used = -INFINITY, l = 0.0f;
    for (int t = 0; t < n_kv_tiles; ++t) {
      const int buf = t & 1;
      // alpha one tile ahead: store tile t + 1 (fetched last iteration), fetch tile t + 2
      if (t + 1 < n_kv_tiles) sm.al[(t + 1) % 3][tid >> 7][tid & (TILE - 1)] = a_next;
      if (t + 2 < n_kv_tiles) a_next = alpha_of(t + 2);
      const float* akt = sm.al[t % 3][0] + hc;
      const float* avt = sm.al[t % 3][1] + hc;
      wait(&sm.bar_s, t & 1);
      ptx::tc_fence_after();
      // pass 1: x = S alpha^K over this thread's 64 tokens (masked), partial row maximum
      const int lim = last - t * TILE - hc;                 // tokens i <= lim are attended
      float x[64];
      {
        uint32_t s0[32], s1[32];
        ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc, s0);
        ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc + 32, s1);
        ptx::tmem_ld_wait();
        ptx::tmem_regs_ready(s0);
        ptx::tmem_regs_ready(s1);
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&sm.sfree);         // this warp's part of S(t) read out
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          x[i] = __uint_as_float(s0[i]) * akt[i];
          x[32 + i] = __uint_as_float(s1[i]) * akt[32 + i];
        }
      }
      const bool full = __all_sync(0xffffffffu, lim >= 63);
      if (!full) {
#pragma unroll
        for (int i = 0; i < 64; ++i) x[i] = i <= lim ? x[i] : -INFINITY;
      }
      float mt = -INFINITY;
#pragma unroll
      for (int i = 0; i < 64; ++i) mt = fmaxf(mt, x[i]);
      sm.xch[buf][half][r] = mt;
      softmax_sync();                                       // partial maxima exchanged
      mt = fmaxf(sm.xch[buf][0][r], sm.xch[buf][1][r]) * rsr;
      const bool need = mt > m_used + kLazyLog2;
      if (__any_sync(0xffffffffu, need && t > 0)) {         // rescale this half of O once PV(t - 1) is done
        wait(&sm.ofree[buf ^ 1], ((t - 1) >> 1) & 1);
        ptx::tc_fence_after();
        const float c = need ? (m_used == -INFINITY ? 0.0f : ex2(m_used - mt)) : 1.0f;
#pragma unroll 1
        for (int ch = 0; ch < 2; ++ch) {
          uint32_t o[32];
          ptx::tmem_ld_32raw(tmem + lane_base + kColO + hc + 32 * ch, o);
          ptx::tmem_ld_wait();
          ptx::tmem_regs_ready(o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * c);
          ptx::tmem_st32(tmem + lane_base + kColO + hc + 32 * ch, o);
        }
      }
      if (need) {
        l = m_used == -INFINITY ? 0.0f : l * ex2(m_used - mt);
        m_used = mt;
      }
      // pass 2: P' = 2^(x rs - m) alpha^V, f16 pairs into P' buffer `buf` once PV(t - 2) has read it
      if (t >= 2) {
        wait(&sm.ofree[buf], ((t - 2) >> 1) & 1);
        ptx::tc_fence_after();
      }
      {
        const float msub = m_used == -INFINITY ? 0.0f : m_used;
        uint32_t pw[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float e0 = ex2(fmaf(x[2 * i], rsr, -msub)), e1 = ex2(fmaf(x[2 * i + 1], rsr, -msub));
          l += e0 + e1;
          pw[i] = pack_h2(e0 * avt[2 * i], e1 * avt[2 * i + 1]);
        }
        ptx::tmem_st32(tmem + lane_base + kColP + 64 * buf + 32 * half, pw);
      }
      ptx::tmem_wait_st();
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&sm.pready);
    }
    if (n_kv_tiles > 0) wait(&sm.ofree[(n_kv_tiles - 1) & 1], ((n_kv_tiles - 1) >> 1) & 1);
    ptx::tc_fence_after();
    // ---- o_hat = f^V O / l, hi / lo bf16 in slots 0 / 1; U_V (rows = dim, K = channel) hi / lo
    // in slots 2 / 3
    softmax_sync();                                       // every warp is past its last maximum exchange
    sm.xch[0][half][r] = l;
    softmax_sync();
    const float lt = sm.xch[0][0][r] + sm.xch[0][1][r];
    {
      const float il = lt > 0.0f ? 1.0f / lt : 0.0f;
      uint32_t o0[32], o1[32];
      ptx::tmem_ld_32raw(tmem + lane_base + kColO + hc, o0);
      ptx::tmem_ld_32raw(tmem + lane_base + kColO + hc + 32, o1);
      ptx::tmem_ld_wait();
      ptx::tmem_regs_ready(o0);
      ptx::tmem_regs_ready(o1);
      const float* fv = a.f + sv * D + hc;
#pragma unroll
      for (int g8 = 0; g8 < 8; ++g8) {
        float u[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int i = 8 * g8 + j;
          const float ov = __uint_as_float(i < 32 ? o0[i & 31] : o1[i & 31]);
          u[j] = lt > 0.0f ? ov * il * fv[i] : 0.0f;
        }
        store_split_bf16(pj + sw128_off(r, hc + 8 * g8), u, 2);
      }
    }
    const float* uv = a.u32 + static_cast<size_t>(sv) * D * D;
    for (int g = tid; g < D * 16; g += kTSoftmax) {
      const int d = g >> 4, k8 = (g & 15) * 8;
      const float4 u0 = *reinterpret_cast<const float4*>(uv + d * D + k8);
      const float4 u1 = *reinterpret_cast<const float4*>(uv + d * D + k8 + 4);
      const float u[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
      store_split_bf16(pj + 2 * kTOp + sw128_off(d, k8), u, 2);
    }
  }
  ptx::fence_proxy_async_smem();
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  // ---- out = o_hat U_V^T = hi.hi + hi.lo + lo.hi
  if (tid == kTCtl) {
#pragma unroll 1
    for (int pr = 0; pr < 3; ++pr) {
      const uint32_t as = pr == 2 ? 1u : 0u, bs = pr == 1 ? 3u : 2u;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t off = (kk >> 2) * kTAtom + (kk & 3) * 32;
        ptx::umma_bf16(tmem + kColS, ptx::sdesc_kmajor_sw128(pj_a + as * kTOp + off),
                       ptx::sdesc_kmajor_sw128(pj_a + bs * kTOp + off), kIdescBB, (pr | kk) ? 1u : 0u);
      }
    }
    ptx::umma_commit(&sm.bar_p);
  }
  if (softmax) {
    wait(&sm.bar_p, 1);
    ptx::tc_fence_after();
    uint32_t o0[32], o1[32];
    ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc, o0);
    ptx::tmem_ld_32raw(tmem + lane_base + kColS + hc + 32, o1);
    ptx::tmem_ld_wait();
    ptx::tmem_regs_ready(o0);
    ptx::tmem_regs_ready(o1);
    if (R < n_rows) {
      const int qi = R / G, qh2 = head * G + R % G;
      float4* dst =
          reinterpret_cast<float4*>(a.out + ((static_cast<size_t>(b) * a.n_q + qi) * a.n_q_heads + qh2) * D + hc);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        dst[i] = make_float4(__uint_as_float(o0[4 * i]), __uint_as_float(o0[4 * i + 1]), __uint_as_float(o0[4 * i + 2]),
                             __uint_as_float(o0[4 * i + 3]));
        dst[8 + i] = make_float4(__uint_as_float(o1[4 * i]), __uint_as_float(o1[4 * i + 1]),
                                 __uint_as_float(o1[4 * i + 2]), __uint_as_float(o1[4 * i + 3]));
      }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

}  // namespace

size_t prefill_workspace(int batch, int n_kv, int n_ctx) {
  const size_t pad = (static_cast<size_t>(n_ctx) + TILE - 1) / TILE * TILE;
  return static_cast<size_t>(batch) * n_kv * 2 * pad * D * sizeof(__half);
}

cudaError_t launch_codes(const Plan& plan, int layer, const void* cache, int batch, int n_ctx, int max_tokens,
                         void* ws, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  PrefillArgs a{};
  a.words = static_cast<const uint32_t*>(cache);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.codes = static_cast<__half*>(ws);
  a.f = plan.dev.f;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.entry = plan.dev.entry;
  a.chan_ent = plan.dev.chan_ent;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.n_ctx = n_ctx;
  a.n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  a.n_tiles = g.n_tiles;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  a.err = plan.dev.err;
  if (plan.n_words > 32) return cudaErrorNotSupported;
  aatc_prefill_codes_kernel<<<dim3(a.n_ctx_pad / TILE, a.n_kv * 2, batch), TILE, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_prefill(const Plan& plan, int layer, const void* q, int q_start, int n_q, const void* cache,
                           int batch, int n_ctx, int max_tokens, float* out, void* ws, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  PrefillArgs a;
  a.words = static_cast<const uint32_t*>(cache);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = out;
  a.codes = static_cast<__half*>(ws);
  a.u32 = plan.dev.u32;
  a.u32t = plan.dev.u32t;
  a.f = plan.dev.f;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.entry = plan.dev.entry;
  a.chan_ent = plan.dev.chan_ent;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.n_q_heads = plan.dims.n_q_heads;
  a.group = a.n_q_heads / a.n_kv;
  a.q_start = q_start;
  a.n_q = n_q;
  a.n_ctx = n_ctx;
  a.n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  a.n_tiles = g.n_tiles;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  a.err = plan.dev.err;
  if (plan.n_words > 32) return cudaErrorNotSupported;
  aatc_prefill_codes_kernel<<<dim3(a.n_ctx_pad / TILE, a.n_kv * 2, batch), TILE, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // one 2D map over the whole codes workspace: rows of 128 f16 (a key token, or a value channel
  // of a 128-token tile), box 64 x 128
  alignas(64) unsigned char tmap[128];
  e = make_tensor_map_2d(tmap, true, ws, D, static_cast<uint64_t>(batch) * a.n_kv * 2 * a.n_ctx_pad, D * 2, 64, TILE);
  if (e != cudaSuccess) return e;
  const size_t smem = sizeof(PrefillTcSmem) + 1024;
  e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_prefill_tc_kernel), smem);
  if (e != cudaSuccess) return e;
  const int n_rows = n_q * a.group;
  aatc_prefill_tc_kernel<<<dim3((n_rows + kTRows - 1) / kTRows, a.n_kv, batch), kTThreads, smem, st>>>(
      *reinterpret_cast<const CUtensorMap*>(tmap), a);
  return cudaGetLastError();
}

}  // namespace aatc
