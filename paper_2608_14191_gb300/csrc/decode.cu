// AATC decode attention over the packed cache, the dequantization test hook, and the
// uncompressed bf16 reference decode (Def. sdpa with one query row; Algorithm 1
// "Reconstruct", "softmax", "Output" lines, computed without rebuilding the keys).
//
// Split-K over the context (flash-decoding): one CTA per (split, kv-head, sequence) computes,
// for the G query heads of its GQA group,
//   phase 1  scores s_{g,t} = alpha^K_t * sum_c q'_{g,c} code^K_{t,c}   (thread = token),
//            with q' = (U_K^T q) * f^K * log2(e) / sqrt(128) folded once per CTA,
//   phase 2  split max m_g, p = 2^(s - m_g), l_g = sum p, P' = p * alpha^V_t,
//   phase 3  acc_{g,c} = sum_t P'_{g,t} code^V_{t,c}   (thread = 4 channels x 1/4 of the tokens),
// and writes (acc, m, l).  The combine kernel merges the splits by log-sum-exp, applies f^V and
// the one inverse value transform out = U_V o_hat.
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>

#include "aatc_internal.h"

namespace aatc {
namespace {

constexpr int kThreads = 128;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Block-wide max / sum of GP values per thread (128 threads).
template <int GP, bool kMax>
__device__ __forceinline__ void block_reduce(float (&v)[GP], float* scratch /* [4][GP] */) {
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float w = __shfl_xor_sync(0xffffffffu, v[g], o);
      v[g] = kMax ? fmaxf(v[g], w) : v[g] + w;
    }
  const int warp = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int g = 0; g < GP; ++g) scratch[warp * GP + g] = v[g];
  __syncthreads();
#pragma unroll
  for (int g = 0; g < GP; ++g) {
    float r = scratch[g];
#pragma unroll
    for (int w = 1; w < 4; ++w) r = kMax ? fmaxf(r, scratch[w * GP + g]) : r + scratch[w * GP + g];
    v[g] = r;
  }
  __syncthreads();
}

// ---------------------------------------------------------------- packed-cache decode
//
// Tensor-core formulation (mma.sync m16n8k16, fp16 operands, fp32 accumulate):
//   scores:  A = folded query q'_c 2^shift per record entry, split hi (rows g) / lo (rows g+8),
//            B = record digits / bits of 8 tokens (each fragment register: one shift + mask of a
//            packed word, then subtracting the 1024 magic), accumulated over the record words.
//   values:  A = probabilities P' = p alpha^V split hi / lo, B = value digits / bits of 16 tokens
//            from the pair-interleaved value words, one n-tile per 8 record entries.
// Token order inside a 16-token group g16 (both products): k = 2i <-> token i, k = 2i+1 <->
// token i+8 for i < 8.  Score n-tile A holds k 0..7, n-tile B k 8..15.

struct DecodeArgs {
  const uint32_t* words;   // cache word region (this layer)
  const float* alpha;      // cache alpha region
  const __nv_bfloat16* q;  // [batch][HQ][128]
  float* ws;               // [batch][HQ][n_splits][n_entries + 3]
  float* out;              // [batch][HQ][128]
  const float* u32;        // plan: [S][128 dim][128 ch]
  const float* u32t;       // plan: [S][128 ch][128 dim]
  const float* f;          // plan: [S][128]
  const ChanEnc* enc;      // plan: [S][128] (offsets 2^(b-1))
  const StreamLayout* lay; // plan: [S]
  const short* entry;      // plan: [S][n_entries]
  const short* chan_ent;   // plan: [S][128][8]
  int* err;
  uint4* qfrag;            // workspace: score A fragments [batch][n_kv][ks_stride]
  float* qcorr;            // workspace: offset corrections [batch][n_kv][8]
  int layer, n_kv, n_q, group, n_ctx, n_tiles, n_words, n_entries, n_splits, split_len, ks_stride, pstride;
};

__device__ __forceinline__ uint32_t hsub_magic(uint32_t x) {
  // x holds two 16-bit fields (1024 + v) as fp16 bit patterns; returns the fp16 pair (v_lo, v_hi)
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(x), "r"(0x64006400u));
  return r;
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__device__ __forceinline__ void mma_16816(float (&c)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}

// 2^x with the hardware approximation (relative error ~2^-22; -inf -> 0)
__device__ __forceinline__ float fast_exp2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// fp32 -> (hi, lo) fp16 pair with hi + lo = v to ~2^-22 relative
__device__ __forceinline__ void split_hi_lo(float v, float& hi, float& lo) {
  hi = __half2float(__float2half_rn(v));
  lo = v - hi;
}

constexpr int kGroups = TILE / 16;        // 16-token groups per tile
constexpr int kWarps = kThreads / 32;

// shared-memory carve-up of the split kernel (32-bit words)
struct SplitLayout {
  int cg, red, run, afrag, pfrag, kw, vw, ak, av, n_words_total;
  __host__ __device__ SplitLayout(int n_ks, int W) {
    int o = 0;
    cg = o;    o += MAX_GROUP;                 // offset corrections
    red = o;   o += 3 * kWarps * MAX_GROUP;    // per-warp max / sum p / sum P'
    run = o;   o += 3 * MAX_GROUP;             // running m, l, S'
    o = (o + 3) & ~3;
    afrag = o; o += n_ks * 32 * 4;             // uint4 per (k-step, lane)
    pfrag = o; o += kGroups * MAX_GROUP * 16;  // half2 (hi, lo) of P' per (group, query, slot)
    kw = o;    o += 2 * W * TILE;              // two stages of key words
    vw = o;    o += 2 * W * TILE;              // two stages of value words
    ak = o;    o += 2 * TILE;
    av = o;    o += 2 * TILE;
    n_words_total = o;
  }
};

// Per call, per (sequence, kv-head): folded query q'_{g,c} = (U_K^T q_g)_c f_c log2(e)/sqrt(128),
// the offset corrections C_g = sum_c q'_{g,c} 2^(b_c-1), and the score A fragments: for each
// k-step and lane, slot k -> record entry (c, shift) -> q'_c 2^shift as fp16 hi (rows g) / lo
// (rows g+8).  512 threads: four quarters of the input dimension per channel.
constexpr int kQThreads = 512;

__global__ void __launch_bounds__(kQThreads)
    aatc_decode_query_kernel(const DecodeArgs a) {
  __shared__ float qf[MAX_GROUP][D];
  __shared__ float part[4][MAX_GROUP][D];
  __shared__ float qc[MAX_GROUP][D];
  __shared__ float credw[kQThreads / 32][MAX_GROUP];
  const int head = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int G = a.group;
  const int sk = (a.layer * a.n_kv + head) * 2;
  for (int i = tid; i < MAX_GROUP * D; i += kQThreads) {
    const int gq = i / D, d = i % D;
    qf[gq][d] = gq < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + gq) * D + d]) : 0.0f;
  }
  __syncthreads();
  {
    const int c = tid & (D - 1), qd = tid >> 7;
    const float* uk = a.u32 + static_cast<size_t>(sk) * D * D + static_cast<size_t>(32 * qd) * D + c;
    float u[32];
#pragma unroll
    for (int d = 0; d < 32; ++d) u[d] = uk[d * D];
    float acc[MAX_GROUP];
#pragma unroll
    for (int gq = 0; gq < MAX_GROUP; ++gq) {
      acc[gq] = 0.0f;
#pragma unroll
      for (int d = 0; d < 32; ++d) acc[gq] = fmaf(u[d], qf[gq][32 * qd + d], acc[gq]);
      part[qd][gq][c] = acc[gq];
    }
  }
  __syncthreads();
  if (tid < D) {
    const int c = tid;
    const float fk = a.f[sk * D + c] * (kLog2e * 0.08838834764831845f);   // 1/sqrt(128)
    const float off = a.enc[sk * D + c].off;
    float cr[MAX_GROUP];
#pragma unroll
    for (int gq = 0; gq < MAX_GROUP; ++gq) {
      const float v = (part[0][gq][c] + part[1][gq][c] + part[2][gq][c] + part[3][gq][c]) * fk;
      qc[gq][c] = v;
      cr[gq] = v * off;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cr[gq] += __shfl_xor_sync(0xffffffffu, cr[gq], o);
    }
    if ((tid & 31) == 0)
#pragma unroll
      for (int gq = 0; gq < MAX_GROUP; ++gq) credw[tid >> 5][gq] = cr[gq];
  }
  __syncthreads();
  if (tid < MAX_GROUP)
    a.qcorr[(static_cast<size_t>(b) * a.n_kv + head) * MAX_GROUP + tid] =
        credw[0][tid] + credw[1][tid] + credw[2][tid] + credw[3][tid];
  const StreamLayout lk = a.lay[sk];
  const int n2w = lk.n2 / 16, n_ks = n2w + 2 * ((lk.n1 + 31) / 32);
  const short* ent = a.entry + static_cast<size_t>(sk) * a.n_entries;
  uint4* dst = a.qfrag + (static_cast<size_t>(b) * a.n_kv + head) * a.ks_stride;
  for (int i = tid; i < n_ks * 32; i += kQThreads) {
    const int ks = i >> 5, ln = i & 31, gq = ln >> 2, tq = ln & 3;
    int fld[4];                                   // fields for k = 2t, 2t+1, 2t+8, 2t+9
    int ebase;
    if (ks < n2w) {
      ebase = 16 * ks;
      fld[0] = tq; fld[1] = tq + 8; fld[2] = tq + 4; fld[3] = tq + 12;
    } else {
      const int r = ks - n2w, h8 = 8 * (r & 1);
      ebase = lk.n2 + 32 * (r >> 1);
      fld[0] = tq + h8; fld[1] = tq + 16 + h8; fld[2] = tq + 4 + h8; fld[3] = tq + 20 + h8;
    }
    float hi[4], lo[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = ebase + fld[j];
      const int ce = (e < lk.n2 + lk.n1) ? ent[e] : -1;
      const float coef = (ce >= 0 && gq < G) ? ldexpf(qc[gq][ce & 0xFF], ce >> 8) : 0.0f;
      split_hi_lo(coef, hi[j], lo[j]);
    }
    dst[i] = make_uint4(pack_half2(hi[0], hi[1]), pack_half2(lo[0], lo[1]), pack_half2(hi[2], hi[3]),
                        pack_half2(lo[2], lo[3]));
  }
}

// Value n-tiles of one record word: a D2 word gives two (fields 0-7 from the low-half lane,
// fields 8-15 from the high-half lane, shift 2g), a D1 word four (low/high lane x shift g, g+8).
template <int WPW, int GP>
__global__ void __launch_bounds__(kThreads)
    aatc_decode_split_kernel(const DecodeArgs a) {
  extern __shared__ __align__(16) uint32_t smw[];
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;                       // mma fragment coordinates
  const int G = a.group;
  const int sk = (a.layer * a.n_kv + head) * 2, sv = sk + 1;   // key / value streams
  const StreamLayout lk = a.lay[sk], lv = a.lay[sv];
  const int W = a.n_words;
  const int n2w_k = lk.n2 / 16, n1w_k = (lk.n1 + 31) / 32;
  const int n_ks = n2w_k + 2 * n1w_k;
  const int n2w_v = lv.n2 / 16, nw_v = n2w_v + (lv.n1 + 31) / 32;
  const SplitLayout L(n_ks, W);
  float* cg = reinterpret_cast<float*>(smw + L.cg);
  float* red = reinterpret_cast<float*>(smw + L.red);          // [3][kWarps][8]
  float* run = reinterpret_cast<float*>(smw + L.run);          // [3][8]: m, l, S'
  uint4* afrag = reinterpret_cast<uint4*>(smw + L.afrag);
  uint32_t* pfrag = smw + L.pfrag;
  uint32_t* kw = smw + L.kw;
  uint32_t* vw = smw + L.vw;
  float* ak = reinterpret_cast<float*>(smw + L.ak);
  float* av = reinterpret_cast<float*>(smw + L.av);

  const int t_begin = split * a.split_len;
  const int t_end = min(a.n_ctx, t_begin + a.split_len);
  const int n_tiles_split = (t_end - t_begin + TILE - 1) / TILE;
  const int tile0 = t_begin / TILE;
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * W * TILE;
  const size_t bk = (static_cast<size_t>(b) * a.n_kv + head) * 2;   // cache stream of the keys
  const uint32_t* kwords = a.words + bk * stream_words;
  const uint32_t* vwords = a.words + (bk + 1) * stream_words;
  const float* kalpha = a.alpha + bk * a.n_tiles * TILE;
  const float* valpha = a.alpha + (bk + 1) * a.n_tiles * TILE;

  auto stage = [&](int tile, int buf) {
    const int chunks = W * (TILE / 4);
    const uint32_t* sk_ = kwords + static_cast<size_t>(tile) * W * TILE;
    const uint32_t* sv_ = vwords + static_cast<size_t>(tile) * W * TILE;
    for (int i = tid; i < chunks; i += kThreads) {
      cp_async16(kw + buf * W * TILE + 4 * i, sk_ + 4 * i);
      cp_async16(vw + buf * W * TILE + 4 * i, sv_ + 4 * i);
    }
    if (tid < TILE / 4) cp_async16(ak + buf * TILE + 4 * tid, kalpha + tile * TILE + 4 * tid);
    else if (tid < TILE / 2) cp_async16(av + buf * TILE + 4 * (tid - TILE / 4), valpha + tile * TILE + 4 * (tid - TILE / 4));
    cp_async_commit();
  };
  stage(tile0, 0);

  // ---- prologue: score A fragments and offset corrections of this (sequence, kv-head), built
  // once per call by aatc_decode_query_kernel
  {
    const uint4* qsrc = a.qfrag + (static_cast<size_t>(b) * a.n_kv + head) * a.ks_stride;
    for (int i = tid; i < n_ks * 32; i += kThreads) cp_async16(afrag + i, qsrc + i);
    cp_async_commit();
    if (tid < MAX_GROUP) {
      cg[tid] = a.qcorr[(static_cast<size_t>(b) * a.n_kv + head) * MAX_GROUP + tid];
      run[tid] = -INFINITY;            // m
      run[8 + tid] = 0.0f;             // l
      run[16 + tid] = 0.0f;            // S'
    }
    for (int i = tid; i < kGroups * MAX_GROUP * 16; i += kThreads) pfrag[i] = 0u;   // rows g >= G stay 0
    cp_async_wait_all();
    __syncthreads();
  }

  // value words of this warp (contiguous) and their n-tile accumulators
  const int vw0 = warp * nw_v / kWarps, vw1 = (warp + 1) * nw_v / kWarps;
  float acc[WPW][4][4];
#pragma unroll
  for (int i = 0; i < WPW; ++i)
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int r = 0; r < 4; ++r) acc[i][q][r] = 0.0f;
  const float c0 = cg[g];

  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage(tile0 + ti + 1, buf ^ 1);
    const uint32_t* kt = kw + buf * W * TILE;
    const uint32_t* vt = vw + buf * W * TILE;
    const int tbase = (tile0 + ti) * TILE;

    // ---- scores: this warp's groups 2 warp, 2 warp + 1 as four n-tiles of 8 tokens
    float sc[4][4];
    int tok[4];
#pragma unroll
    for (int n = 0; n < 4; ++n) {
      tok[n] = 16 * (2 * warp + (n >> 1)) + (g & 1 ? 8 : 0) + (g >> 1) + 4 * (n & 1);   // column g's token
#pragma unroll
      for (int r = 0; r < 4; ++r) sc[n][r] = 0.0f;
    }
    for (int wd = 0; wd < n2w_k; ++wd) {
      const uint4 af = afrag[wd * 32 + lane];
#pragma unroll
      for (int n = 0; n < 4; ++n) {
        const uint32_t x = kt[wd * TILE + tok[n]];
        mma_16816(sc[n], af, hsub_magic(((x >> (2 * t)) & 0x00030003u) | 0x64006400u),
                  hsub_magic(((x >> (2 * t + 8)) & 0x00030003u) | 0x64006400u));
      }
    }
    for (int w1 = 0; w1 < n1w_k; ++w1) {
      const int wd = n2w_k + w1;
      const uint4 af0 = afrag[(n2w_k + 2 * w1) * 32 + lane];
      const uint4 af1 = afrag[(n2w_k + 2 * w1 + 1) * 32 + lane];
#pragma unroll
      for (int n = 0; n < 4; ++n) {
        const uint32_t x = kt[wd * TILE + tok[n]];
        mma_16816(sc[n], af0, hsub_magic(((x >> t) & 0x00010001u) | 0x64006400u),
                  hsub_magic(((x >> (t + 4)) & 0x00010001u) | 0x64006400u));
        mma_16816(sc[n], af1, hsub_magic(((x >> (t + 8)) & 0x00010001u) | 0x64006400u),
                  hsub_magic(((x >> (t + 12)) & 0x00010001u) | 0x64006400u));
      }
    }
    // lane holds query g, columns 2t (token ta) and 2t+1 (token ta + 8) of each n-tile
    float s8[4][2];
    float mloc = -INFINITY;
#pragma unroll
    for (int n = 0; n < 4; ++n) {
      const int ta = 16 * (2 * warp + (n >> 1)) + t + 4 * (n & 1);
      const float sa = ak[buf * TILE + ta] * (sc[n][0] + sc[n][2] - c0);
      const float sb = ak[buf * TILE + ta + 8] * (sc[n][1] + sc[n][3] - c0);
      s8[n][0] = (g < G && tbase + ta < t_end) ? sa : -INFINITY;
      s8[n][1] = (g < G && tbase + ta + 8 < t_end) ? sb : -INFINITY;
      mloc = fmaxf(mloc, fmaxf(s8[n][0], s8[n][1]));
    }
    mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, 1));
    mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, 2));
    if (t == 0) red[warp * 8 + g] = mloc;
    __syncthreads();
    const float m_old = run[g];
    float m_new = m_old;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) m_new = fmaxf(m_new, red[w * 8 + g]);
    const float corr = m_old == -INFINITY ? 0.0f : fast_exp2(m_old - m_new);
    // probabilities, P' = p alpha^V, partial sums, and the P' fragments for the value product
    float lsum = 0.0f, ssum = 0.0f;
#pragma unroll
    for (int gg = 0; gg < 2; ++gg) {
      float pv[4];
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          const int n = 2 * gg + h;
          const int tk = 16 * (2 * warp + gg) + t + 4 * h + 8 * cc;
          const float p = s8[n][cc] == -INFINITY ? 0.0f : fast_exp2(s8[n][cc] - m_new);
          const float pp = p * av[buf * TILE + tk];
          lsum += p;
          ssum += pp;
          pv[2 * h + cc] = pp;                 // slot 4t + {0: token t, 1: t+8, 2: t+4, 3: t+12}
        }
      if (g < G) {
        uint4 pk;
        float hi, lo;
        split_hi_lo(pv[0], hi, lo); pk.x = pack_half2(hi, lo);
        split_hi_lo(pv[1], hi, lo); pk.y = pack_half2(hi, lo);
        split_hi_lo(pv[2], hi, lo); pk.z = pack_half2(hi, lo);
        split_hi_lo(pv[3], hi, lo); pk.w = pack_half2(hi, lo);
        *reinterpret_cast<uint4*>(pfrag + ((2 * warp + gg) * MAX_GROUP + g) * 16 + 4 * t) = pk;
      }
    }
    lsum += __shfl_xor_sync(0xffffffffu, lsum, 1);
    lsum += __shfl_xor_sync(0xffffffffu, lsum, 2);
    ssum += __shfl_xor_sync(0xffffffffu, ssum, 1);
    ssum += __shfl_xor_sync(0xffffffffu, ssum, 2);
    if (t == 0) {
      red[(kWarps + warp) * 8 + g] = lsum;
      red[(2 * kWarps + warp) * 8 + g] = ssum;
    }
    __syncthreads();
    if (warp == 0 && t == 0) {
      float l = 0.0f, sp = 0.0f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        l += red[(kWarps + w) * 8 + g];
        sp += red[(2 * kWarps + w) * 8 + g];
      }
      run[g] = m_new;
      run[8 + g] = run[8 + g] * corr + l;
      run[16 + g] = run[16 + g] * corr + sp;
    }

    // ---- values: this warp's record words over the 8 groups of the tile
#pragma unroll
    for (int i = 0; i < WPW; ++i)
#pragma unroll
      for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int r = 0; r < 4; ++r) acc[i][q][r] *= corr;
#pragma unroll 2
    for (int g16 = 0; g16 < kGroups; ++g16) {
      const uint4 pf = *reinterpret_cast<const uint4*>(pfrag + (g16 * MAX_GROUP + g) * 16 + 4 * t);
      uint4 af;
      af.x = __byte_perm(pf.x, pf.y, 0x5410);      // hi of tokens t, t+8
      af.y = __byte_perm(pf.x, pf.y, 0x7632);      // lo
      af.z = __byte_perm(pf.z, pf.w, 0x5410);      // hi of tokens t+4, t+12
      af.w = __byte_perm(pf.z, pf.w, 0x7632);      // lo
#pragma unroll
      for (int i = 0; i < WPW; ++i) {
        const int wd = vw0 + i;
        if (wd < vw1) {
          const uint4 vx = *reinterpret_cast<const uint4*>(vt + wd * TILE + 16 * g16 + 4 * t);
          if (wd < n2w_v) {
            mma_16816(acc[i][0], af, hsub_magic(((vx.x >> (2 * g)) & 0x00030003u) | 0x64006400u),
                      hsub_magic(((vx.z >> (2 * g)) & 0x00030003u) | 0x64006400u));
            mma_16816(acc[i][1], af, hsub_magic(((vx.y >> (2 * g)) & 0x00030003u) | 0x64006400u),
                      hsub_magic(((vx.w >> (2 * g)) & 0x00030003u) | 0x64006400u));
          } else {
            mma_16816(acc[i][0], af, hsub_magic(((vx.x >> g) & 0x00010001u) | 0x64006400u),
                      hsub_magic(((vx.z >> g) & 0x00010001u) | 0x64006400u));
            mma_16816(acc[i][1], af, hsub_magic(((vx.x >> (g + 8)) & 0x00010001u) | 0x64006400u),
                      hsub_magic(((vx.z >> (g + 8)) & 0x00010001u) | 0x64006400u));
            mma_16816(acc[i][2], af, hsub_magic(((vx.y >> g) & 0x00010001u) | 0x64006400u),
                      hsub_magic(((vx.w >> g) & 0x00010001u) | 0x64006400u));
            mma_16816(acc[i][3], af, hsub_magic(((vx.y >> (g + 8)) & 0x00010001u) | 0x64006400u),
                      hsub_magic(((vx.w >> (g + 8)) & 0x00010001u) | 0x64006400u));
          }
        }
      }
    }
  }
  cp_async_wait_all();
  __syncthreads();

  // ---- partials: value sums per record entry, then m, l, S'
  if (g < G) {
    float* dst = a.ws + ((static_cast<size_t>(b) * a.n_q + head * G + g) * a.n_splits + split) * a.pstride;
#pragma unroll
    for (int i = 0; i < WPW; ++i) {
      const int wd = vw0 + i;
      if (wd < vw1) {
        const int ebase = wd < n2w_v ? 16 * wd : lv.n2 + 32 * (wd - n2w_v);
        const int nq = wd < n2w_v ? 2 : 4;
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (q < nq) {
            dst[ebase + 8 * q + 2 * t] = acc[i][q][0] + acc[i][q][2];
            dst[ebase + 8 * q + 2 * t + 1] = acc[i][q][1] + acc[i][q][3];
          }
      }
    }
    if (warp == 0 && t == 0) {
      dst[a.n_entries] = run[g];
      dst[a.n_entries + 1] = run[8 + g];
      dst[a.n_entries + 2] = run[16 + g];
    }
  }
}

// Merge the splits of one (sequence, query head) by log-sum-exp, rebuild channel sums from the
// record entries (o_c = sum_e 2^shift_e O_e - 2^(b_c-1) S'), scale by f^V / l, apply U_V.
// The partials of all splits are staged in shared memory with 16-byte loads first.
constexpr int kCThreads = 256;

__global__ void __launch_bounds__(kCThreads)
    aatc_decode_combine_kernel(const DecodeArgs a) {
  extern __shared__ __align__(16) float cs[];
  const int stride = a.pstride;                      // multiple of 4
  float* part = cs;                                  // [n_splits][stride]
  float* wsp = part + a.n_splits * stride;           // [n_splits] split weights
  float* oe = wsp + ((a.n_splits + 3) & ~3);         // [n_entries]
  float* ohat = oe + a.n_entries;                    // [128]
  float* ut_s = ohat + D;                            // [128][128] U_V^T of this kv-head
  __shared__ float red[2][kCThreads / 32];
  __shared__ float lsum[2];
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int head = j / a.group;
  const int sv = (a.layer * a.n_kv + head) * 2 + 1;
  const float4* src = reinterpret_cast<const float4*>(a.ws + (static_cast<size_t>(b) * a.n_q + j) * a.n_splits * stride);
  const int n4 = a.n_splits * stride / 4;
  float4* p4 = reinterpret_cast<float4*>(part);
  for (int i = tid; i < n4; i += kCThreads) cp_async16(p4 + i, src + i);
  const float4* us = reinterpret_cast<const float4*>(a.u32t + static_cast<size_t>(sv) * D * D);
  for (int i = tid; i < D * D / 4; i += kCThreads) cp_async16(reinterpret_cast<float4*>(ut_s) + i, us + i);
  cp_async_commit();
  cp_async_wait_all();
  __syncthreads();
  // split weights 2^(m_s - M): every thread scans the split maxima (few dozen)
  float m = -INFINITY;
  for (int s = 0; s < a.n_splits; ++s) m = fmaxf(m, part[s * stride + a.n_entries]);
  if (tid < a.n_splits) wsp[tid] = exp2f(part[tid * stride + a.n_entries] - m);
  for (int s = tid + kCThreads; s < a.n_splits; s += kCThreads) wsp[s] = exp2f(part[s * stride + a.n_entries] - m);
  __syncthreads();
  if (tid < 64) {
    float l = 0.0f, sp = 0.0f;
    for (int s = tid; s < a.n_splits; s += 64) {
      l += part[s * stride + a.n_entries + 1] * wsp[s];
      sp += part[s * stride + a.n_entries + 2] * wsp[s];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      l += __shfl_xor_sync(0xffffffffu, l, o);
      sp += __shfl_xor_sync(0xffffffffu, sp, o);
    }
    if ((tid & 31) == 0) {
      red[0][tid >> 5] = l;
      red[1][tid >> 5] = sp;
    }
  }
  const StreamLayout lv = a.lay[sv];
  const int n_used = lv.n2 + lv.n1;
  for (int e = tid; e < n_used; e += kCThreads) {
    float acc = 0.0f;
    for (int s = 0; s < a.n_splits; ++s) acc = fmaf(part[s * stride + e], wsp[s], acc);
    oe[e] = acc;
  }
  __syncthreads();
  if (tid == 0) {
    lsum[0] = red[0][0] + red[0][1];
    lsum[1] = red[1][0] + red[1][1];
  }
  __syncthreads();
  if (tid < D) {
    const int c = tid;
    const short* ce = a.chan_ent + (static_cast<size_t>(sv) * D + c) * 8;
    const short* ent = a.entry + static_cast<size_t>(sv) * a.n_entries;
    float o = 0.0f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int e = ce[k];
      if (e >= 0) o += ldexpf(oe[e], ent[e] >> 8);
    }
    o -= a.enc[sv * D + c].off * lsum[1];
    ohat[c] = o * a.f[sv * D + c] / lsum[0];
  }
  __syncthreads();
  {
    // out[d] = sum_c U_V[d][c] ohat[c]; two threads per output dimension
    const int d = tid & (D - 1), half = tid >> 7;
    float o = 0.0f;
#pragma unroll 16
    for (int c = half * 64; c < half * 64 + 64; ++c) o = fmaf(ut_s[c * D + d], ohat[c], o);
    if (half) oe[d] = o;
    __syncthreads();
    if (!half) a.out[(static_cast<size_t>(b) * a.n_q + j) * D + d] = o + oe[d];
  }
}

// ---------------------------------------------------------------- bf16 reference decode
struct Bf16Args {
  const __nv_bfloat16* k;  // [batch][max_tokens][n_kv][128]
  const __nv_bfloat16* v;
  const __nv_bfloat16* q;  // [batch][n_q][128]
  float* ws;
  int n_kv, n_q, group, n_ctx, max_tokens, n_splits, split_len;
};

__device__ __forceinline__ void bf16x8_to_f32(const uint4 r, float* o) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[2 * i] = __uint_as_float(w[i] << 16);
    o[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

template <int GP>
__global__ void __launch_bounds__(kThreads)
    aatc_bf16_split_kernel(const Bf16Args a) {
  extern __shared__ __align__(16) float sm[];
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int G = a.group;
  constexpr int kRow = D + 8;                              // padded bf16 row (272 B)
  float* qs = sm;                                          // [128][GP]
  float* red = qs + D * GP;                                // [32]
  float* sc = red + 32;                                    // [split_len][GP]
  __nv_bfloat16* kt = reinterpret_cast<__nv_bfloat16*>(sc + a.split_len * GP);   // [2][128][kRow]
  float* accs = reinterpret_cast<float*>(kt + 2 * TILE * kRow);                  // [4][GP][128]
  const int t_begin = split * a.split_len;
  const int t_end = min(a.n_ctx, t_begin + a.split_len);
  const int n_tiles_split = (t_end - t_begin + TILE - 1) / TILE;
  const float scale = kLog2e * 0.08838834764831845f;
  for (int i = tid; i < GP * D; i += kThreads) {
    const int g = i / D, d = i % D;
    qs[d * GP + g] =
        g < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + g) * D + d]) * scale : 0.0f;
  }
  auto stage = [&](const __nv_bfloat16* base, int tile, int buf) {
    __nv_bfloat16* dst = kt + buf * TILE * kRow;
    for (int i = tid; i < TILE * 16; i += kThreads) {
      const int r = i >> 4, ch = i & 15;
      int t = tile * TILE + r;
      t = min(t, a.n_ctx - 1);                             // clamp padding rows to a valid token
      cp_async16(dst + r * kRow + ch * 8, base + ((static_cast<size_t>(b) * a.max_tokens + t) * a.n_kv + head) * D + ch * 8);
    }
    cp_async_commit();
  };
  const int tile0 = t_begin / TILE;
  stage(a.k, tile0, 0);
  __syncthreads();
  float mloc[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) mloc[g] = -INFINITY;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage(a.k, tile0 + ti + 1, buf ^ 1);
    const __nv_bfloat16* row = kt + buf * TILE * kRow + tid * kRow;
    float s[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) s[g] = 0.0f;
    for (int d0 = 0; d0 < D; d0 += 8) {
      float kv[8];
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(row + d0), kv);
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int g4 = 0; g4 < GP; g4 += 4) {
          const float4 qv = *reinterpret_cast<const float4*>(qs + (d0 + i) * GP + g4);
          s[g4] = fmaf(qv.x, kv[i], s[g4]);
          s[g4 + 1] = fmaf(qv.y, kv[i], s[g4 + 1]);
          s[g4 + 2] = fmaf(qv.z, kv[i], s[g4 + 2]);
          s[g4 + 3] = fmaf(qv.w, kv[i], s[g4 + 3]);
        }
    }
    const int t = (tile0 + ti) * TILE + tid;
    float* out = sc + (ti * TILE + tid) * GP;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float v = t < t_end ? s[g] : -INFINITY;
      out[g] = v;
      mloc[g] = fmaxf(mloc[g], v);
    }
  }
  cp_async_wait_all();
  __syncthreads();
  block_reduce<GP, true>(mloc, red);
  stage(a.v, tile0, 0);
  float lsum[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) lsum[g] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    float* p = sc + (ti * TILE + tid) * GP;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float e = exp2f(p[g] - mloc[g]);
      lsum[g] += e;
      p[g] = e;
    }
  }
  block_reduce<GP, false>(lsum, red);
  const int dg = tid & 31, tq = tid >> 5;
  float acc[GP][4];
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[g][i] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage(a.v, tile0 + ti + 1, buf ^ 1);
    const int tend = min(TILE, t_end - (tile0 + ti) * TILE);
    for (int tt = tq; tt < tend; tt += 4) {
      const uint2 r = *reinterpret_cast<const uint2*>(kt + buf * TILE * kRow + tt * kRow + dg * 4);
      const float vv[4] = {__uint_as_float(r.x << 16), __uint_as_float(r.x & 0xFFFF0000u),
                           __uint_as_float(r.y << 16), __uint_as_float(r.y & 0xFFFF0000u)};
      const float* p = sc + (ti * TILE + tt) * GP;
#pragma unroll
      for (int g4 = 0; g4 < GP; g4 += 4) {
        const float4 pv = *reinterpret_cast<const float4*>(p + g4);
        const float pg[4] = {pv.x, pv.y, pv.z, pv.w};
#pragma unroll
        for (int gg = 0; gg < 4; ++gg)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[g4 + gg][i] = fmaf(pg[gg], vv[i], acc[g4 + gg][i]);
      }
    }
  }
  cp_async_wait_all();
  __syncthreads();
#pragma unroll
  for (int g = 0; g < GP; ++g)
    *reinterpret_cast<float4*>(accs + (tq * GP + g) * D + dg * 4) = make_float4(acc[g][0], acc[g][1], acc[g][2], acc[g][3]);
  __syncthreads();
  for (int g = 0; g < G; ++g) {
    const float v = accs[(0 * GP + g) * D + tid] + accs[(1 * GP + g) * D + tid] + accs[(2 * GP + g) * D + tid] +
                    accs[(3 * GP + g) * D + tid];
    float* dst = a.ws + ((static_cast<size_t>(b) * a.n_q + head * G + g) * a.n_splits + split) * (D + 3);
    dst[tid] = v;
    if (tid == 0) {
      dst[D] = mloc[g];
      dst[D + 1] = lsum[g];
      dst[D + 2] = 0.0f;
    }
  }
}

// Log-sum-exp merge of bf16-reference partials (identity output transform).
__global__ void __launch_bounds__(kThreads)
    aatc_plain_combine_kernel(const float* ws, int n_splits, int n_q, float* out) {
  __shared__ float red[8];
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int stride = D + 3;
  const float* src = ws + (static_cast<size_t>(b) * n_q + j) * n_splits * stride;
  float m = -INFINITY;
  for (int s = tid; s < n_splits; s += kThreads) m = fmaxf(m, src[s * stride + D]);
  float mv[1] = {m};
  block_reduce<1, true>(mv, red);
  m = mv[0];
  float l = 0.0f;
  for (int s = tid; s < n_splits; s += kThreads) l += src[s * stride + D + 1] * exp2f(src[s * stride + D] - m);
  float lv[1] = {l};
  block_reduce<1, false>(lv, red);
  float acc = 0.0f;
  for (int s = 0; s < n_splits; ++s) acc += src[s * stride + tid] * exp2f(src[s * stride + D] - m);
  out[(static_cast<size_t>(b) * n_q + j) * D + tid] = acc / lv[0];
}

// Dequantization hook: thread per (sequence, token, stream) of the requested range; rebuilds
// each stored value from its record entries and returns fl32(code * fl32(alpha * f_c)).
__global__ void aatc_dequant_kernel(const uint32_t* words, const float* alpha, const StreamLayout* lays,
                                    const short* entry, const float* f, int layer, int n_kv, int batch, int t0,
                                    int n, int n_tiles, int n_words, int n_entries, float* out) {
  const long idx = static_cast<long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const long total = static_cast<long>(batch) * n * n_kv * 2;
  if (idx >= total) return;
  const int kind = static_cast<int>(idx % 2);
  const int head = static_cast<int>((idx / 2) % n_kv);
  const int i = static_cast<int>((idx / (2 * n_kv)) % n);
  const int b = static_cast<int>(idx / (2L * n_kv * n));
  const int t = t0 + i;
  const size_t cs = (static_cast<size_t>(b) * n_kv + head) * 2 + kind;
  const uint32_t* tile = words + cs * n_tiles * n_words * TILE + static_cast<size_t>(t / TILE) * n_words * TILE;
  const int tt = t % TILE;
  int lane_lo = tt, lane_hi = tt, half = 0;
  if (kind == 1) {
    const int j = tt & 15, pr = j & 7;
    lane_lo = 16 * (tt >> 4) + 4 * (pr & 3) + 2 * (pr >> 2);
    lane_hi = lane_lo + 1;
    half = j >> 3;
  }
  auto rec_word = [&](int w) -> uint32_t {
    if (kind == 0) return tile[static_cast<size_t>(w) * TILE + tt];
    const uint32_t lo = (tile[static_cast<size_t>(w) * TILE + lane_lo] >> (16 * half)) & 0xFFFFu;
    const uint32_t hi = (tile[static_cast<size_t>(w) * TILE + lane_hi] >> (16 * half)) & 0xFFFFu;
    return lo | (hi << 16);
  };
  const int s = (layer * n_kv + head) * 2 + kind;
  const StreamLayout ly = lays[s];
  const short* ent = entry + static_cast<size_t>(s) * n_entries;
  uint32_t u[D];
  for (int c = 0; c < D; ++c) u[c] = 0u;
  for (int e = 0; e < ly.n2 + ly.n1; ++e) {
    const int ce = ent[e];
    uint32_t v;
    if (e < ly.n2) {
      v = (rec_word(e >> 4) >> (2 * (e & 15))) & 3u;
    } else {
      const int e1 = e - ly.n2;
      v = (rec_word(ly.n2 / 16 + (e1 >> 5)) >> (e1 & 31)) & 1u;
    }
    u[ce & 0xFF] |= v << (ce >> 8);
  }
  const float at = alpha[cs * n_tiles * TILE + t];
  float* o = out + idx * D;
  for (int c = 0; c < D; ++c) {
    const float fc = f[s * D + c];
    float v = 0.0f;
    if (fc != 0.0f) {
      int nb = 0;
      for (int e = 0; e < ly.n2 + ly.n1; ++e)
        if ((ent[e] & 0xFF) == c) nb = max(nb, (ent[e] >> 8) + (e < ly.n2 ? 2 : 1));
      const int code = static_cast<int>(u[c]) - (1 << (nb - 1));
      v = __fmul_rn(static_cast<float>(code), __fmul_rn(at, fc));
    }
    o[c] = v;
  }
}

template <int WPW, int GP>
cudaError_t launch_split_t(const DecodeArgs& a, int batch, size_t smem, cudaStream_t st) {
  static size_t smem_set = 0;                                  // raise the opt-in limit only when needed
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(aatc_decode_split_kernel<WPW, GP>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  aatc_decode_split_kernel<WPW, GP><<<dim3(a.n_splits, a.n_kv, batch), kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

template <int GP>
cudaError_t launch_split_g(const DecodeArgs& a, int batch, int wpw, size_t smem, cudaStream_t st) {
  if (wpw <= 3) return launch_split_t<3, GP>(a, batch, smem, st);
  if (wpw <= 4) return launch_split_t<4, GP>(a, batch, smem, st);
  return launch_split_t<8, GP>(a, batch, smem, st);
}

template <int GP>
cudaError_t launch_bf16_split(const Bf16Args& a, int batch, cudaStream_t st) {
  const size_t smem = 4 * (static_cast<size_t>(D) * GP + 32 + static_cast<size_t>(a.split_len) * GP + 4 * GP * D) +
                      2 * static_cast<size_t>(TILE) * (D + 8) * 2;
  static size_t smem_set = 0;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(aatc_bf16_split_kernel<GP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  aatc_bf16_split_kernel<GP><<<dim3(a.n_splits, a.n_kv, batch), kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                          int max_tokens, float* out, void* ws, const DecodeSplit& sp, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  DecodeArgs a;
  a.words = static_cast<const uint32_t*>(cache);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.ws = static_cast<float*>(ws);
  a.out = out;
  a.u32 = plan.dev.u32;
  a.u32t = plan.dev.u32t;
  a.f = plan.dev.f;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.entry = plan.dev.entry;
  a.chan_ent = plan.dev.chan_ent;
  a.err = plan.dev.err;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.n_q = plan.dims.n_q_heads;
  a.group = a.n_q / a.n_kv;
  a.n_ctx = n_ctx;
  a.n_tiles = g.n_tiles;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  a.n_splits = sp.n_splits;
  a.split_len = sp.split_len;
  // largest key k-step count and value word count over the layer's streams
  int n_ks = 1, nw_v = 1;
  for (int h = 0; h < a.n_kv; ++h) {
    const StreamLayout& lk = plan.layout[(layer * a.n_kv + h) * 2];
    const StreamLayout& lv = plan.layout[(layer * a.n_kv + h) * 2 + 1];
    n_ks = std::max(n_ks, lk.n2 / 16 + 2 * ((lk.n1 + 31) / 32));
    nw_v = std::max(nw_v, lv.n2 / 16 + (lv.n1 + 31) / 32);
  }
  const DecodeWs wsl = decode_ws_layout(batch, a.n_q, a.n_kv, plan.n_entries, plan.n_words, sp);
  a.pstride = wsl.pstride;
  a.ks_stride = wsl.ks_stride;
  a.qfrag = reinterpret_cast<uint4*>(static_cast<char*>(ws) + wsl.qfrag_off);
  a.qcorr = reinterpret_cast<float*>(static_cast<char*>(ws) + wsl.qcorr_off);
  aatc_decode_query_kernel<<<dim3(a.n_kv, batch), kQThreads, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const SplitLayout L(n_ks, plan.n_words);
  const size_t smem = 4 * static_cast<size_t>(L.n_words_total);
  const int wpw = (nw_v + kWarps - 1) / kWarps;
  if (wpw > 8) return cudaErrorNotSupported;
  e = a.group <= 4 ? launch_split_g<4>(a, batch, wpw, smem, st) : launch_split_g<8>(a, batch, wpw, smem, st);
  if (e != cudaSuccess) return e;
  const size_t csmem =
      4 * (static_cast<size_t>(a.n_splits) * a.pstride + ((a.n_splits + 3) & ~3) + plan.n_entries + D + D * D);
  static size_t csmem_set = 0;
  if (csmem > 48 * 1024 && csmem > csmem_set) {
    e = cudaFuncSetAttribute(aatc_decode_combine_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(csmem));
    if (e != cudaSuccess) return e;
    csmem_set = csmem;
  }
  aatc_decode_combine_kernel<<<dim3(a.n_q, batch), kCThreads, csmem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_dequant(const Plan& plan, int layer, const void* cache, int batch, int t0, int n, int max_tokens,
                           float* out, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  const long total = static_cast<long>(batch) * n * plan.dims.n_kv_heads * 2;
  const int threads = 128;
  const long blocks = (total + threads - 1) / threads;
  aatc_dequant_kernel<<<static_cast<unsigned>(blocks), threads, 0, st>>>(
      static_cast<const uint32_t*>(cache), reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems),
      plan.dev.lay, plan.dev.entry, plan.dev.f, layer, plan.dims.n_kv_heads, batch, t0, n, g.n_tiles, plan.n_words,
      plan.n_entries, out);
  return cudaGetLastError();
}

cudaError_t launch_bf16_decode(const void* K, const void* V, const void* q, int batch, int n_ctx, int max_tokens,
                               int n_kv, int n_q, float* out, void* ws, const DecodeSplit& sp, cudaStream_t st) {
  Bf16Args a;
  a.k = static_cast<const __nv_bfloat16*>(K);
  a.v = static_cast<const __nv_bfloat16*>(V);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.ws = static_cast<float*>(ws);
  a.n_kv = n_kv;
  a.n_q = n_q;
  a.group = n_q / n_kv;
  a.n_ctx = n_ctx;
  a.max_tokens = max_tokens;
  a.n_splits = sp.n_splits;
  a.split_len = sp.split_len;
  cudaError_t e = a.group <= 4 ? launch_bf16_split<4>(a, batch, st) : launch_bf16_split<8>(a, batch, st);
  if (e != cudaSuccess) return e;
  aatc_plain_combine_kernel<<<dim3(n_q, batch), kThreads, 0, st>>>(a.ws, a.n_splits, n_q, out);
  return cudaGetLastError();
}

}  // namespace aatc

// ------------------------------------------------------------------ decode without a workspace
// For callers that cannot allocate device memory at call time (see aatc_decode_attention_noalloc
// in aatc.h): the split partials live in one fixed array of this file, reserved on every device
// that loads the library.  Host code must not use the array's name as an address; the device
// address is looked up once per device with cudaGetSymbolAddress.
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[AATC_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mutex;
void* g_noalloc_address[kMaxDevices] = {};

}  // namespace

extern "C" aatc_status_t aatc_decode_attention_noalloc(aatc_plan_t p, int32_t layer, const void* q,
                                                       const void* cache, int32_t batch, int32_t n_ctx,
                                                       int32_t max_tokens, float* out, void* stream) {
  using namespace aatc;
  Plan* plan = plan_from_handle(p);
  if (!plan || !q || !cache || !out || layer < 0 || layer >= plan->dims.n_layers || batch < 1 || n_ctx < 1 ||
      max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (n_ctx > max_tokens) return AATC_ERR_CAPACITY;
  if (plan->dims.n_q_heads / plan->dims.n_kv_heads > MAX_GROUP) return AATC_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(cache) & 15u) != 0) return AATC_ERR_INVALID_ARG;
  const DecodeSplit sp = decode_split(batch, plan->dims.n_kv_heads, n_ctx, plan->num_sms);
  if (decode_workspace(batch, plan->dims.n_q_heads, plan->dims.n_kv_heads, plan->n_entries, plan->n_words, sp) >
      AATC_NOALLOC_SCRATCH_BYTES)
    return AATC_ERR_WORKSPACE;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return status_from_cuda(e);
  if (dev < 0 || dev >= kMaxDevices) return AATC_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_address[dev]) {
      e = cudaGetSymbolAddress(&g_noalloc_address[dev], g_noalloc_scratch);
      if (e != cudaSuccess) {
        g_noalloc_address[dev] = nullptr;
        return status_from_cuda(e);
      }
    }
    scratch = g_noalloc_address[dev];
  }
  return status_from_cuda(launch_decode(*plan, layer, q, cache, batch, n_ctx, max_tokens, out, scratch, sp,
                                        static_cast<cudaStream_t>(stream)));
}
