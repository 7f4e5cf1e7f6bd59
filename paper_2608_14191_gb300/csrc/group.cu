// Decode attention over head-group streams (Sec. 5 Step 1, remark on multi-head attention: the
// g_h kv-heads of a group share one transform; Def. sdpa per query head, Algorithm 1's
// reconstruct / attend / output lines in the transformed space).
//
// A group stream of n = 128 g_h channels is stored as g_h slice streams in the per-kv-head slots
// (slice s = storage channels s, s + g_h, ...), one alpha per token.  Query head j of the group
// (kv-head block m = j / group) sees the embedded query q~ (q at block m, zeros elsewhere):
//   score_t = (U_K^T q~) . h_hat_t / sqrt(128) = alpha_t sum_c q'_c f_c code_tc,
//   out     = rows of block m of U_V applied to sum_t p_t h_hat^V_t.
// Three launches per call:
//   query  per (query row < 16, slice, group, sequence): q'' = (U_K^T q~) f log2(e) / sqrt(128)
//          over the slice's 128 channels, the slice's scale and part of the offset correction, and
//          the row's words of the slice's score A fragments (entry order of its key records)
//   attn   per (split, group, sequence), 8 warps: the slices' record words are the operands of
//          mma.sync m16n8k16 f16 (a digit or bit masked into a 16-bit half is the subnormal
//          digit 2^-24), rows = the group's <= 16 query heads: scores summed over every slice
//          and corrected by the stored-value offsets, online softmax with the exponent of
//          alpha^V folded into the running maximum (P' = 2^(s - m) alpha^V < 2), value entry sums
//          per slice, channel sums at the end of the split
//   merge  per (query head, slice, group, sequence): log-sum-exp over the splits, o_hat = f^V O
//          over the slice's channels and its part of U_V[block m rows] o_hat; the last slice to
//          arrive adds the parts in slice order and divides by l
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "aatc_internal.h"
#include "ptx.cuh"

namespace aatc {
namespace {

constexpr float kGLog2e = 1.4426950408889634f;
constexpr int kGAThreads = 256;                  // 8 warps; each also runs the softmax of 16 tokens

struct GroupDecodeArgs {
  const float* alpha;        // cache alpha region [b][n_kv][K|V][n_tiles * 128]
  const __nv_bfloat16* q;    // [b][H_q][128]
  const float* uk;           // plan: U_K of every (layer, group), [n dim][n channel]
  const float* uvt;          // plan: U_V^T, [n channel][n dim]
  const float* f;            // plan: [slot][128] f_c
  uint32_t* qfrag;           // workspace: score A fragments [b][n_groups][hi | lo][g_h][ks_max][32][4] (f16 pairs)
  float* qsc;                // workspace: [b][n_groups][16][g_h][scale, C part] of each query row and slice
  float* outp;               // workspace: [b][n_groups][16][g_h][128] per-slice output partials
  int* ticket;               // workspace: [b][n_groups][16] merge arrivals (zeroed by the query kernel)
  float* part;               // workspace: split partials [b][n_groups][nq][n_splits][n + 4]
  float* out;                // [b][H_q][128]
  const uint32_t* words;     // cache word region (the digit kernel reads the records directly)
  const short* entry;        // plan: [slot][n_entries] (channel | shift << 8), -1 padded
  const ChanEnc* enc;        // plan: [slot][128] (offset 2^(b-1) of each stored value)
  const StreamLayout* lay;   // plan: [slot]
  int layer, n_kv, gh, n_groups, group, nq, n, n_q_heads, n_ctx, n_ctx_pad, n_tiles, n_splits;
  int n_words, n_entries, ks_max, stages;    // ks_max: k-steps of the widest slice; stages: ring depth
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}
__device__ __forceinline__ float fexp2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// f16 hi / lo parts of x and y, packed as (x, y) pairs
__device__ __forceinline__ void split2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x, y);
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(x - hf.x, y - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Per (query row i < 16, slice s, group, sequence), 512 threads = 128 channels x 4 quarters of the
// 128 query dims; slice channel c is slice-major channel j' = 128 s + c:
//   q''_j' = (U_K^T q~)_j' f_j' log2(e) / sqrt(128)   (zero for rows i >= nq),
//   scale  = 2^(ceil(log2 max_c |q''| 2^(b - 1)) - 14) so that every A entry q'' 2^shift / scale of
//            the slice is below 2^14,
//   C_s    = sum_c q''_j' 2^(b_j' - 1) (the slice's part of the key codes' stored-value offsets),
// and row i's words of the slice's score A fragments: for k-step ks and lane column t, the f16
// pairs (k 2t, 2t + 1) and (k 2t + 8, 2t + 9) of q'' 2^shift 2^-p / scale over the k-step's entries
// (p = 2t for base-4 words, t for bit words: the position at which the digit kernel leaves the
// lane's fields), hi and lo parts.
constexpr int kGQThreads = 512;
__global__ void __launch_bounds__(kGQThreads) aatc_group_query_kernel(const GroupDecodeArgs a) {
  __shared__ float qv[D];
  __shared__ float part[4][D];
  __shared__ float qsm[D];
  __shared__ float redx[4], redc[4];
  __shared__ float s_scale;
  const int i = blockIdx.x, s = blockIdx.y % a.gh, g = blockIdx.y / a.gh, b = blockIdx.z, tid = threadIdx.x;
  const int c = tid & (D - 1), dq = tid >> 7;
  const bool live = i < a.nq;
  const int m = i / a.group, hq = g * a.nq + i;
  const size_t bg = static_cast<size_t>(b) * a.n_groups + g;
  if (s == 0 && tid == 0) a.ticket[bg * 16 + i] = 0;
  if (live && tid < D) qv[tid] = __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q_heads + hq) * D + tid]);
  __syncthreads();
  const int pslot = (a.layer * a.n_kv + g * a.gh + s) * 2;   // plan slot of the slice's keys
  if (live) {
    const float* u = a.uk + (static_cast<size_t>(a.layer) * a.n_groups + g) * a.n * a.n +
                     static_cast<size_t>(m * D + 32 * dq) * a.n + s * D + c;
    float x[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) x[k] = u[static_cast<size_t>(k) * a.n];   // 32 loads in flight per thread
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int k = 0; k < 32; ++k) acc[k & 3] = fmaf(x[k], qv[32 * dq + k], acc[k & 3]);
    part[dq][c] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
  }
  __syncthreads();
  if (tid < D) {
    const float qj = live ? ((part[0][c] + part[1][c]) + (part[2][c] + part[3][c])) * a.f[pslot * D + c] *
                                (kGLog2e * 0.08838834764831845f)
                          : 0.0f;
    qsm[c] = qj;
    const float off = a.enc[pslot * D + c].off;
    float mx = fabsf(qj) * off, cc = qj * off;
    for (int o = 16; o > 0; o >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      cc += __shfl_xor_sync(0xffffffffu, cc, o);
    }
    if ((tid & 31) == 0) {
      redx[tid >> 5] = mx;
      redc[tid >> 5] = cc;
    }
  }
  __syncthreads();
  if (tid == 0) {
    const float mt = fmaxf(fmaxf(redx[0], redx[1]), fmaxf(redx[2], redx[3]));
    int ex = 0;
    if (mt > 0.0f) frexpf(mt, &ex);
    s_scale = ldexpf(1.0f, ex - 14);
    a.qsc[((bg * 16 + i) * a.gh + s) * 2] = s_scale;
    a.qsc[((bg * 16 + i) * a.gh + s) * 2 + 1] = (redc[0] + redc[1]) + (redc[2] + redc[3]);
  }
  __syncthreads();
  const float inv = 1.0f / s_scale;
  const size_t fw = static_cast<size_t>(a.gh) * a.ks_max * 128;   // u32 words of one (hi or lo) table
  uint32_t* fh = a.qfrag + bg * 2 * fw;
  uint32_t* fl = fh + fw;
  const StreamLayout& ly = a.lay[pslot];
  const int n2 = ly.n2, ne = ly.n2 + ly.n1, n2w = n2 / 16, nks = n2w + 2 * ((ly.n1 + 31) / 32);
  const short* et = a.entry + static_cast<size_t>(pslot) * a.n_entries;
  for (int item = tid; item < a.ks_max * 8; item += kGQThreads) {
    const int ks = item >> 3, tt = (item >> 1) & 3, kp = item & 1;
    int e0 = -1, e1 = -1;                          // entries at k = 2t + 8 kp and 2t + 8 kp + 1
    float lsc = 0.0f;
    if (ks < n2w) {                                // base-4 word: fields t, t + 8 | t + 4, t + 12
      e0 = 16 * ks + tt + 4 * kp;
      e1 = e0 + 8;
      lsc = ldexpf(1.0f, -2 * tt);
    } else if (ks < nks) {                         // bit word, half s2: bits t, t + 16 | t + 4, t + 20
      const int uw = (ks - n2w) >> 1, s2 = (ks - n2w) & 1;
      e0 = n2 + 32 * uw + 8 * s2 + tt + 4 * kp;
      e1 = e0 + 16;
      lsc = ldexpf(1.0f, -tt);
    }
    const int c0 = e0 >= 0 && e0 < ne ? et[e0] : -1, c1 = e1 >= 0 && e1 < ne ? et[e1] : -1;
    const float v0 = c0 >= 0 ? qsm[c0 & 0xFF] * ldexpf(lsc, (c0 >> 8) & 15) * inv : 0.0f;
    const float v1 = c1 >= 0 ? qsm[c1 & 0xFF] * ldexpf(lsc, (c1 >> 8) & 15) * inv : 0.0f;
    uint32_t hi, lo;
    split2(v0, v1, hi, lo);
    // A fragment registers: a0 = row r (k 2t..), a1 = row r + 8, a2 = row r (k 2t + 8..), a3 = row r + 8
    const size_t idx = ((static_cast<size_t>(s) * a.ks_max + ks) * 32 + (i & 7) * 4 + tt) * 4 + kp * 2 + (i >> 3);
    fh[idx] = hi;
    fl[idx] = lo;
  }
}

// ---------------------------------------------------------------- digit-operand split attention
// The slices' record words are the tensor-core operands themselves (no unpacked codes): a base-4
// digit (or a single bit) masked into a 16-bit half is the subnormal f16 value d 2^(p - 24), p its
// bit position in the half; the power 2^p is folded into the other operand's scale.
//   chunks: per tile, the key words of all g_h slices, then their value words (cp.async ring)
//   scores: warp (slice sl, part) over its slice's k-steps and 8 (g_h = 4) or 4 (g_h = 2)
//           token n-tiles: A = q''_c 2^shift per entry (rows = queries, hi / lo, lane t's columns
//           scaled by 2^-2t for D2 words, 2^-t for D1 words), B = the tokens' fields masked in
//           place; the slice partials meet in shared memory and are summed per token, then
//           raw = sum q'' u, s = alpha^K (raw - C) with C = sum_c q''_c 2^(b_c - 1)
//   values: warp (slice sl, part) owns the 8-entry tiles part, part + 8 / g_h, ... of slice sl:
//           A = P' (queries x 16 tokens, hi / lo, loaded once per k-step), B = the entries'
//           fields of those tokens from the quad-interleaved value slots (byte permute + mask);
//           the entry sums become channel sums o_c = sum_e 2^(shift - p) O_e - 2^(b_c - 1) S'
//           (S' = the represented sum of P') through shared-memory adds at the end of the split.
constexpr int kGRS = TILE + 8;                   // padded row stride of the per-slice score partials

struct GroupDigitSmem {
  int qfh, qfl, pfh, pfl, ring, red, offs, info, misc, total, chunk_words;
  __host__ __device__ GroupDigitSmem(int gh, int ks_max, int n_words, int stages) {
    chunk_words = n_words * TILE;                 // one slice, one kind, one tile
    const int qf = gh * ks_max * 32 * 16, pf = (TILE / 16) * 32 * 16;
    const int rw = stages * gh * chunk_words * 4, qc = 16 * D * gh * 4;
    int o = 0;
    qfh = o;   o += qf;                           // [slice][k-step][lane] uint4, hi parts
    qfl = o;   o += qf;                           //   lo parts
    pfh = o;   o += pf;                           // [k-step][lane] uint4, hi parts of P'
    pfl = o;   o += pf;
    ring = o;  o += rw > qc ? rw : qc;            // record chunks; channel sums at the end
    red = o;   o += gh * 16 * kGRS * 4;           // [slice][query][token] score partials
    offs = o;  o += D * gh * 4;                   // stored-value offsets 2^(b-1) of the values
    info = o;  o += 16 * gh;                      // [slice][K|V] (n2, n1)
    misc = o;  o += 16 * 4 * (gh + 5) + 3 * 8 * 16 * 4;
    total = o;
  }
};

template <int GH, int NPW>
__global__ void __launch_bounds__(kGAThreads, 1) aatc_group_digit_kernel(const GroupDecodeArgs a) {
  constexpr int N = D * GH, WPS = 8 / GH, NTK = TILE / (8 * WPS);   // warps per slice, key n-tiles per warp
  extern __shared__ __align__(128) unsigned char smb[];
  const GroupDigitSmem L(GH, a.ks_max, a.n_words, a.stages);
  uint4* qfh = reinterpret_cast<uint4*>(smb + L.qfh);
  uint4* qfl = reinterpret_cast<uint4*>(smb + L.qfl);
  uint4* pfh = reinterpret_cast<uint4*>(smb + L.pfh);
  uint4* pfl = reinterpret_cast<uint4*>(smb + L.pfl);
  uint32_t* ring = reinterpret_cast<uint32_t*>(smb + L.ring);
  float* red = reinterpret_cast<float*>(smb + L.red);
  float* offv = reinterpret_cast<float*>(smb + L.offs);
  int* info = reinterpret_cast<int*>(smb + L.info);
  float* qsl = reinterpret_cast<float*>(smb + L.misc);   // [16][g_h] slice scales x 2^24
  float* mrow = qsl + 16 * GH;
  float* lrow = mrow + 16;
  float* srow = lrow + 16;                        // S' of each query
  float* rscale = srow + 16;
  float* corr = rscale + 16;                      // C of each query
  float* redm = corr + 16;                        // [8][16]
  float* reds = redm + 8 * 16;                    // [8][16]
  float* redp = reds + 8 * 16;                    // [8][16]
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, gq = lane >> 2, t = lane & 3;
  const int ws = warp / WPS, wsub = warp % WPS;   // this warp's slice and its part of the slice
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE;
  const int tile_lo = static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const size_t slot0 = static_cast<size_t>(b) * a.n_kv + static_cast<size_t>(g) * GH;   // cache slot of slice 0
  const float* kalpha = a.alpha + (slot0 * 2) * a.n_tiles * TILE;
  const float* valpha = a.alpha + (slot0 * 2 + 1) * a.n_tiles * TILE;
  const size_t bg = static_cast<size_t>(b) * a.n_groups + g;
  const int pslot0 = (a.layer * a.n_kv + g * GH) * 2;   // plan slot of slice 0, keys (values + 1)
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;

  // ---- the score A fragments (built by the query kernel) by cp.async, with the first ring chunk;
  // the value offsets, the slice layouts and the query scales by plain loads
  {
    const int fw = GH * a.ks_max * 128;
    const uint32_t* fsrc = a.qfrag + bg * 2 * fw;
    uint32_t* fdst = reinterpret_cast<uint32_t*>(qfh);   // hi table, then the lo table (contiguous)
    for (int p = tid * 4; p < 2 * fw; p += kGAThreads * 4) cp_async16(fdst + p, fsrc + p);
  }
  for (int j = tid; j < N; j += kGAThreads) offv[j] = a.enc[(pslot0 + 2 * (j / D) + 1) * D + j % D].off;
  if (tid < 2 * GH) {
    info[2 * tid] = a.lay[pslot0 + tid].n2;
    info[2 * tid + 1] = a.lay[pslot0 + tid].n1;
  }
  if (tid < 16 * GH) qsl[tid] = a.qsc[(bg * 16 * GH + tid) * 2] * 16777216.0f;
  if (tid < 16) {
    float cs = 0.0f;
#pragma unroll
    for (int sl = 0; sl < GH; ++sl) cs += a.qsc[((bg * 16 + tid) * GH + sl) * 2 + 1];
    corr[tid] = cs;
    mrow[tid] = -INFINITY;
    lrow[tid] = 0.0f;
    srow[tid] = 0.0f;
  }
  __syncthreads();
  // ---- this warp's value pairs (8-entry tiles wsub, wsub + WPS, ... of slice ws): word offset of
  // the lane's entry and the in-place mask of its field (bit position p = the entry's shift in its byte)
  const int n2v = info[4 * ws + 2], nev = n2v + info[4 * ws + 3], ntpv = (nev + 7) >> 3;
  const int npv = ntpv > wsub ? min(NPW, (ntpv - wsub + WPS - 1) / WPS) : 0;
  int poff[NPW];
  uint32_t pmask[NPW];
#pragma unroll
  for (int j = 0; j < NPW; ++j) {
    const int e = 8 * (wsub + WPS * j) + gq;
    int widx = 0, qp = 0, sh = 0;
    uint32_t mm = 0;
    if (j < npv && e < n2v) {
      const int f = e & 15;
      widx = e >> 4;
      qp = f >> 2;
      sh = 2 * (f & 3);
      mm = 0x00030003u;
    } else if (j < npv && e < nev) {
      const int e1 = e - n2v, bb = e1 & 31;
      widx = (n2v >> 4) + (e1 >> 5);
      qp = bb >> 3;
      sh = bb & 7;
      mm = 0x00010001u;
    }
    qp = qp == 1 ? 2 : qp == 2 ? 1 : qp;          // quarter slot of the byte within the quad
    poff[j] = widx * TILE + qp + 4 * (t >> 1);
    pmask[j] = mm << sh;
  }
  const uint32_t psel = (2 * (t & 1)) | 0x40u | ((2 * (t & 1) + 1) << 8) | 0x4000u;   // bytes i0, i0 + 1 -> halves

  // ---- record chunks: per tile the key words of slices 0 .. GH-1, then their value words
  const int n_chunks = 2 * (tile_hi - tile_lo);
  const int S = a.stages, cw = L.chunk_words;
  auto issue = [&](int u) {
    if (u < n_chunks) {
      const int tile = tile_lo + (u >> 1), kind = u & 1;
      uint32_t* dst = ring + (u % S) * GH * cw;
#pragma unroll
      for (int sl = 0; sl < GH; ++sl) {
        const uint32_t* src = a.words + ((slot0 + sl) * 2 + kind) * stream_words + static_cast<size_t>(tile) * cw;
        for (int p = tid * 4; p < cw; p += kGAThreads * 4) cp_async16(dst + sl * cw + p, src + p);
      }
    }
    cp_async_commit();
  };
  for (int u = 0; u < S - 1; ++u) issue(u);

  float oacc[NPW][4];
#pragma unroll
  for (int j = 0; j < NPW; ++j)
#pragma unroll
    for (int r = 0; r < 4; ++r) oacc[j][r] = 0.0f;
  const int n2k = info[4 * ws], n2wk = n2k >> 4, n1wk = (info[4 * ws + 1] + 31) >> 5;
  const uint32_t M2 = 0x00030003u << (2 * t), M1 = 0x00010001u << t;
  const int tb = wsub * 8 * NTK, tw = 16 * warp;

  for (int u = 0; u < n_chunks; ++u) {
    issue(u + S - 1);
    if (S == 3) cp_async_wait<2>();
    else cp_async_wait<1>();
    __syncthreads();
    const int tile = tile_lo + (u >> 1);
    const uint32_t* cs = ring + (u % S) * GH * cw + ws * cw;   // this warp's slice
    if ((u & 1) == 0) {
      // ---- slice partial scores of tokens tb .. tb + 8 NTK
      float sacc[NTK][4];
#pragma unroll
      for (int nt = 0; nt < NTK; ++nt)
#pragma unroll
        for (int r = 0; r < 4; ++r) sacc[nt][r] = 0.0f;
      const uint4* qh = qfh + ws * a.ks_max * 32 + lane;
      const uint4* ql = qfl + ws * a.ks_max * 32 + lane;
      for (int w = 0; w < n2wk; ++w) {
        const uint4 ah = qh[w * 32], al = ql[w * 32];
#pragma unroll
        for (int nt = 0; nt < NTK; ++nt) {
          const uint32_t x = cs[w * TILE + tb + 8 * nt + gq];
          const uint32_t b0 = x & M2, b1 = (x >> 8) & M2;
          mma16816(sacc[nt], ah, b0, b1);
          mma16816(sacc[nt], al, b0, b1);
        }
      }
      for (int w = 0; w < n1wk; ++w) {
        const int ks = n2wk + 2 * w;
        const uint4 ah0 = qh[ks * 32], al0 = ql[ks * 32], ah1 = qh[ks * 32 + 32], al1 = ql[ks * 32 + 32];
#pragma unroll
        for (int nt = 0; nt < NTK; ++nt) {
          const uint32_t x = cs[(n2wk + w) * TILE + tb + 8 * nt + gq];
          const uint32_t b0 = x & M1, b1 = (x >> 4) & M1, b2 = (x >> 8) & M1, b3 = (x >> 12) & M1;
          mma16816(sacc[nt], ah0, b0, b1);
          mma16816(sacc[nt], al0, b0, b1);
          mma16816(sacc[nt], ah1, b2, b3);
          mma16816(sacc[nt], al1, b2, b3);
        }
      }
      float* rs = red + ws * 16 * kGRS;
#pragma unroll
      for (int nt = 0; nt < NTK; ++nt) {
        const int col = tb + 8 * nt + 2 * t;
        *reinterpret_cast<float2*>(&rs[gq * kGRS + col]) = make_float2(sacc[nt][0], sacc[nt][1]);
        *reinterpret_cast<float2*>(&rs[(gq + 8) * kGRS + col]) = make_float2(sacc[nt][2], sacc[nt][3]);
      }
      __syncthreads();
      // ---- online softmax of the tile (warp w < 8: tokens 16 w ..), raw = sum_s acc_s 2^24 scale_s - C.
      // Lane (gq, t) holds rows gq, gq + 8 and tokens tw + 8 nt + 2t + {0, 1}; e = s + floor(log2 alpha^V)
      // keeps P' = 2^(e - m) mant(alpha^V) < 2.
      float e[2][4], mant[2][4], lav[2][4];
      if (warp < 8) {
      float sc[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const int col = tw + 8 * nt + 2 * t;
        float2 s0 = make_float2(0.0f, 0.0f), s1 = make_float2(0.0f, 0.0f);
#pragma unroll
        for (int sl = 0; sl < GH; ++sl) {
          const float2 v0 = *reinterpret_cast<const float2*>(&red[(sl * 16 + gq) * kGRS + col]);
          const float2 v1 = *reinterpret_cast<const float2*>(&red[(sl * 16 + gq + 8) * kGRS + col]);
          const float w0 = qsl[gq * GH + sl], w1 = qsl[(gq + 8) * GH + sl];
          s0.x = fmaf(v0.x, w0, s0.x); s0.y = fmaf(v0.y, w0, s0.y);
          s1.x = fmaf(v1.x, w1, s1.x); s1.y = fmaf(v1.y, w1, s1.y);
        }
        sc[nt][0] = s0.x; sc[nt][1] = s0.y; sc[nt][2] = s1.x; sc[nt][3] = s1.y;
      }
      float mx0 = -INFINITY, mx1 = -INFINITY;
      const float c0 = corr[gq], c1 = corr[gq + 8];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int tok = tile * TILE + tw + 8 * nt + 2 * t + (r & 1);
          const int row = r < 2 ? gq : gq + 8;
          const bool ok = tok < a.n_ctx && row < a.nq;
          float ev = -INFINITY, mv = 0.0f, lv = 0.0f;
          if (ok) {
            const float ak = kalpha[tok], avv = valpha[tok];
            const float sv = (sc[nt][r] - (r < 2 ? c0 : c1)) * ak;
            int ex = 0;
            const float fr = frexpf(avv, &ex);
            lv = avv > 0.0f ? static_cast<float>(max(ex - 1, -64)) : -64.0f;
            mv = avv > 0.0f ? fr * 2.0f : 0.0f;
            if (avv > 0.0f && ex - 1 < -64) mv = avv * 18446744073709551616.0f;
            ev = sv + lv;
          }
          e[nt][r] = ev;
          mant[nt][r] = mv;
          lav[nt][r] = lv;
          if (r < 2) mx0 = fmaxf(mx0, ev);
          else mx1 = fmaxf(mx1, ev);
        }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      if (t == 0) {
        redm[warp * 16 + gq] = mx0;
        redm[warp * 16 + gq + 8] = mx1;
      }
      }
      __syncthreads();
      if (tid < 16) {
        float mt = -INFINITY;
#pragma unroll
        for (int w = 0; w < 8; ++w) mt = fmaxf(mt, redm[w * 16 + tid]);
        const float mo = mrow[tid], mn = fmaxf(mo, mt);
        rscale[tid] = mo == -INFINITY ? 0.0f : fexp2(mo - mn);
        mrow[tid] = mn;
      }
      __syncthreads();
      if (warp < 8) {
      const float m0 = mrow[gq], m1r = mrow[gq + 8];
      float ls0 = 0.0f, ls1 = 0.0f, ps0 = 0.0f, ps1 = 0.0f;
      float p[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const float mm = r < 2 ? m0 : m1r;
          const float x = e[nt][r] == -INFINITY ? 0.0f : fexp2(e[nt][r] - mm);
          p[nt][r] = x * mant[nt][r];
          const float l = e[nt][r] == -INFINITY ? 0.0f : x * exp2f(-lav[nt][r]);
          if (r < 2) ls0 += l;
          else ls1 += l;
        }
      uint4 ph, pl;
      split2(p[0][0], p[0][1], ph.x, pl.x);
      split2(p[0][2], p[0][3], ph.y, pl.y);
      split2(p[1][0], p[1][1], ph.z, pl.z);
      split2(p[1][2], p[1][3], ph.w, pl.w);
      pfh[warp * 32 + lane] = ph;
      pfl[warp * 32 + lane] = pl;
      // S': the represented P' (hi + lo) that the value MMAs add
      {
        const __half2* hh = reinterpret_cast<const __half2*>(&ph);
        const __half2* ll = reinterpret_cast<const __half2*>(&pl);
        float2 v;
        v = __half22float2(hh[0]); ps0 += v.x + v.y; v = __half22float2(ll[0]); ps0 += v.x + v.y;
        v = __half22float2(hh[2]); ps0 += v.x + v.y; v = __half22float2(ll[2]); ps0 += v.x + v.y;
        v = __half22float2(hh[1]); ps1 += v.x + v.y; v = __half22float2(ll[1]); ps1 += v.x + v.y;
        v = __half22float2(hh[3]); ps1 += v.x + v.y; v = __half22float2(ll[3]); ps1 += v.x + v.y;
      }
      ls0 += __shfl_xor_sync(0xffffffffu, ls0, 1);
      ls0 += __shfl_xor_sync(0xffffffffu, ls0, 2);
      ls1 += __shfl_xor_sync(0xffffffffu, ls1, 1);
      ls1 += __shfl_xor_sync(0xffffffffu, ls1, 2);
      ps0 += __shfl_xor_sync(0xffffffffu, ps0, 1);
      ps0 += __shfl_xor_sync(0xffffffffu, ps0, 2);
      ps1 += __shfl_xor_sync(0xffffffffu, ps1, 1);
      ps1 += __shfl_xor_sync(0xffffffffu, ps1, 2);
      if (t == 0) {
        reds[warp * 16 + gq] = ls0;
        reds[warp * 16 + gq + 8] = ls1;
        redp[warp * 16 + gq] = ps0;
        redp[warp * 16 + gq + 8] = ps1;
      }
      }
      // value accumulators: rows of D are the queries (c0, c1: row gq; c2, c3: row gq + 8)
      const float r0 = rscale[gq], r1 = rscale[gq + 8];
#pragma unroll
      for (int j = 0; j < NPW; ++j) {
        oacc[j][0] *= r0;
        oacc[j][1] *= r0;
        oacc[j][2] *= r1;
        oacc[j][3] *= r1;
      }
      __syncthreads();
      if (tid < 16) {
        float lt = 0.0f, pt = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          lt += reds[w * 16 + tid];
          pt += redp[w * 16 + tid];
        }
        lrow[tid] = lrow[tid] * rscale[tid] + lt;
        srow[tid] = srow[tid] * rscale[tid] + pt;
      }
    } else {
      // ---- O_e += P' . field_e 2^p over this warp's pairs, P' loaded once per k-step
#pragma unroll
      for (int kt = 0; kt < TILE / 16; ++kt) {
        const uint4 ah = pfh[kt * 32 + lane], al = pfl[kt * 32 + lane];
#pragma unroll
        for (int j = 0; j < NPW; ++j) {
          if (j < npv) {
            const uint32_t x0 = cs[poff[j] + 16 * kt], x1 = cs[poff[j] + 16 * kt + 8];
            const uint32_t b0 = __byte_perm(x0, 0u, psel) & pmask[j], b1 = __byte_perm(x1, 0u, psel) & pmask[j];
            mma16816(oacc[j], ah, b0, b1);
            mma16816(oacc[j], al, b0, b1);
          }
        }
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();
  __syncthreads();

  // ---- entry sums -> channel sums (shared-memory adds), then the split's partials
  float* oc = reinterpret_cast<float*>(ring);     // [16][N]
  for (int i = tid; i < 16 * N; i += kGAThreads) oc[i] = 0.0f;
  __syncthreads();
  {
    const short* et = a.entry + static_cast<size_t>(pslot0 + 2 * ws + 1) * a.n_entries;
#pragma unroll
    for (int j = 0; j < NPW; ++j) {
      if (j >= npv) break;
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int e = 8 * (wsub + WPS * j) + 2 * t + k;   // D column 2t + k
        const int ce = e < nev ? et[e] : -1;
        if (ce < 0) continue;
        const int p = e < n2v ? 2 * (e & 3) : (e - n2v) & 7;   // the field's bit position in its byte
        const float w2 = ldexpf(1.0f, ((ce >> 8) & 15) + 24 - p);   // fields entered as d 2^(p - 24)
        const int jj = ws * D + (ce & 0xFF);
        if (gq < a.nq) atomicAdd(&oc[gq * N + jj], w2 * oacc[j][k]);
        if (gq + 8 < a.nq) atomicAdd(&oc[(gq + 8) * N + jj], w2 * oacc[j][2 + k]);
      }
    }
  }
  __syncthreads();
  const size_t pstride = static_cast<size_t>(N) + 4;
  float* pb = a.part + ((static_cast<size_t>(b) * a.n_groups + g) * a.nq) * a.n_splits * pstride;
  for (int idx = tid; idx < a.nq * N; idx += kGAThreads) {
    const int i = idx / N, j = idx % N;
    pb[(static_cast<size_t>(i) * a.n_splits + split) * pstride + j] = oc[i * N + j] - offv[j] * srow[i];
  }
  if (tid < a.nq) {
    float* d = pb + (static_cast<size_t>(tid) * a.n_splits + split) * pstride + N;
    d[0] = mrow[tid];
    d[1] = lrow[tid];
  }
}

// Per (query head i, slice s, group, sequence), 512 threads: combine the splits (weights
// 2^(m_s - M), l = sum w_s l_s), o_hat_j' = f^V_j' sum_s w_s O_s,j' over the slice's 128 channels
// (4 quarters of the splits), then the slice's part of U_V[block m rows] o_hat (4 quarters of the
// channels).  The CTA that arrives last for (i, group, sequence) adds the g_h parts in slice order
// and divides by l, so the result does not depend on the arrival order.
constexpr int kGMThreads = 512;
__global__ void __launch_bounds__(kGMThreads) aatc_group_merge_kernel(const GroupDecodeArgs a) {
  extern __shared__ float wsp[];                  // w [n_splits]
  __shared__ float red[kGMThreads / 32];
  __shared__ float part[4][D];
  __shared__ float ohat[D];
  __shared__ float s_l;
  __shared__ int s_last;
  const int i = blockIdx.x, s = blockIdx.y % a.gh, g = blockIdx.y / a.gh, b = blockIdx.z, tid = threadIdx.x;
  const int N = a.n, m = i / a.group, c = tid & (D - 1), q4 = tid >> 7;
  const size_t bg = static_cast<size_t>(b) * a.n_groups + g;
  const size_t pstride = static_cast<size_t>(N) + 4;
  const float* pb = a.part + ((bg * a.nq + i) * a.n_splits) * pstride;
  // M = max_s m_s (block reduction), then w_s and l = sum_s w_s l_s
  float mloc = -INFINITY;
  for (int s2 = tid; s2 < a.n_splits; s2 += kGMThreads) mloc = fmaxf(mloc, pb[s2 * pstride + N]);
  for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
  if ((tid & 31) == 0) red[tid >> 5] = mloc;
  __syncthreads();
  float M = -INFINITY;
  for (int w = 0; w < kGMThreads / 32; ++w) M = fmaxf(M, red[w]);
  __syncthreads();
  float lloc = 0.0f;
  for (int s2 = tid; s2 < a.n_splits; s2 += kGMThreads) {
    const float ms = pb[s2 * pstride + N];
    const float w = ms == -INFINITY ? 0.0f : exp2f(ms - M);
    wsp[s2] = w;
    lloc += w * pb[s2 * pstride + N + 1];
  }
  for (int o = 16; o > 0; o >>= 1) lloc += __shfl_xor_sync(0xffffffffu, lloc, o);
  if ((tid & 31) == 0) red[tid >> 5] = lloc;
  __syncthreads();
  if (tid == 0) {
    float l = 0.0f;
    for (int w = 0; w < kGMThreads / 32; ++w) l += red[w];
    s_l = l;
  }
  // o_hat over the slice's channels: quarter q4 takes splits q4, q4 + 4, ...
  {
    const float* pc = pb + s * D + c;
    float o[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    for (int s0 = q4; s0 < a.n_splits; s0 += 4 * 24) {   // 24 loads in flight per thread
      float x[24];
#pragma unroll
      for (int k = 0; k < 24; ++k) x[k] = s0 + 4 * k < a.n_splits ? pc[static_cast<size_t>(s0 + 4 * k) * pstride] : 0.0f;
#pragma unroll
      for (int k = 0; k < 24; ++k)
        if (s0 + 4 * k < a.n_splits) o[k & 3] = fmaf(wsp[s0 + 4 * k], x[k], o[k & 3]);
    }
    part[q4][c] = (o[0] + o[1]) + (o[2] + o[3]);
  }
  __syncthreads();
  if (tid < D) {
    const int slot = (a.layer * a.n_kv + g * a.gh + s) * 2 + 1;
    ohat[c] = ((part[0][c] + part[1][c]) + (part[2][c] + part[3][c])) * a.f[slot * D + c];
  }
  __syncthreads();
  // the slice's part of U_V[block m rows] o_hat: quarter q4 takes channels 32 q4 .. 32 q4 + 31
  {
    const float* u = a.uvt + (static_cast<size_t>(a.layer) * a.n_groups + g) * static_cast<size_t>(N) * N +
                     static_cast<size_t>(s * D + 32 * q4) * N + static_cast<size_t>(m) * D + c;
    float x[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) x[k] = u[static_cast<size_t>(k) * N];   // 32 loads in flight per thread
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int k = 0; k < 32; ++k) acc[k & 3] = fmaf(x[k], ohat[32 * q4 + k], acc[k & 3]);
    part[q4][c] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
  }
  __syncthreads();
  float* op = a.outp + (bg * 16 + i) * a.gh * D;
  if (tid < D) op[s * D + c] = (part[0][c] + part[1][c]) + (part[2][c] + part[3][c]);
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&a.ticket[bg * 16 + i], 1) == a.gh - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < D) {
    float o = 0.0f;
    for (int s2 = 0; s2 < a.gh; ++s2) o += __ldcg(&op[s2 * D + c]);
    a.out[(static_cast<size_t>(b) * a.n_q_heads + g * a.nq + i) * D + c] = o / s_l;
  }
}

int group_splits(const Plan& plan, int batch, int n_ctx) {
  const int tiles = (n_ctx + TILE - 1) / TILE;
  const int units = batch * (plan.dims.n_kv_heads / plan.group_heads);
  return std::max(1, std::min(tiles, std::max(1, plan.num_sms) / std::max(1, units)));
}

struct GroupWs {
  size_t frag_off, qsc_off, outp_off, ticket_off, part_off, bytes;
};
// k-steps (D2 words + 2 x D1 words) of the widest slice stream of `layer` (keys or values)
int group_ks_max(const Plan& plan, int layer) {
  int m = 1;
  for (int h = 0; h < plan.dims.n_kv_heads; ++h)
    for (int kind = 0; kind < 2; ++kind) {
      const StreamLayout& ly = plan.layout[(layer * plan.dims.n_kv_heads + h) * 2 + kind];
      m = std::max(m, ly.n2 / 16 + 2 * ((ly.n1 + 31) / 32));
    }
  return m;
}

GroupWs group_ws_layout(const Plan& plan, int batch, int n_ctx) {
  const int ng = plan.dims.n_kv_heads / plan.group_heads, n = D * plan.group_heads;
  const int nq = plan.dims.n_q_heads / ng;
  int ks = 1;                                     // the widest layer's k-steps size the fragment tables
  for (int l = 0; l < plan.dims.n_layers; ++l) ks = std::max(ks, group_ks_max(plan, l));
  GroupWs w;
  size_t off = 0;
  w.frag_off = off;
  off += static_cast<size_t>(batch) * ng * 2 * plan.group_heads * ks * 128 * 4;
  w.qsc_off = off;
  off += static_cast<size_t>(batch) * ng * 16 * plan.group_heads * 2 * 4;
  w.outp_off = off;
  off += static_cast<size_t>(batch) * ng * 16 * plan.group_heads * D * 4;
  w.ticket_off = off;
  off += static_cast<size_t>(batch) * ng * 16 * 4;
  off = (off + 255) / 256 * 256;
  w.part_off = off;
  off += static_cast<size_t>(batch) * ng * nq * group_splits(plan, batch, n_ctx) * (n + 4) * 4;
  w.bytes = off;
  return w;
}

}  // namespace

size_t group_decode_workspace(const Plan& plan, int batch, int n_ctx) { return group_ws_layout(plan, batch, n_ctx).bytes; }

cudaError_t launch_group_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                                int max_tokens, float* out, void* ws, cudaStream_t st) {
  const int gh = plan.group_heads;
  if (gh != 2 && gh != 4) return cudaErrorNotSupported;
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  const GroupWs wl = group_ws_layout(plan, batch, n_ctx);
  GroupDecodeArgs a;
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.uk = plan.gdev.uk;
  a.uvt = plan.gdev.uvt;
  a.f = plan.dev.f;
  a.qfrag = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + wl.frag_off);
  a.qsc = reinterpret_cast<float*>(static_cast<char*>(ws) + wl.qsc_off);
  a.outp = reinterpret_cast<float*>(static_cast<char*>(ws) + wl.outp_off);
  a.ticket = reinterpret_cast<int*>(static_cast<char*>(ws) + wl.ticket_off);
  a.part = reinterpret_cast<float*>(static_cast<char*>(ws) + wl.part_off);
  a.out = out;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.gh = gh;
  a.n_groups = a.n_kv / gh;
  a.group = plan.dims.n_q_heads / a.n_kv;
  a.nq = gh * a.group;
  a.n = D * gh;
  a.n_q_heads = plan.dims.n_q_heads;
  a.n_ctx = n_ctx;
  a.n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  a.n_tiles = g.n_tiles;
  a.n_splits = group_splits(plan, batch, n_ctx);
  a.words = static_cast<const uint32_t*>(cache);
  a.entry = plan.dev.entry;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  a.ks_max = group_ks_max(plan, layer);
  // value pairs per warp: 8-entry tiles of the widest value slice over the 8 / g_h warps of a slice
  int ntp = 1;
  for (int h = 0; h < a.n_kv; ++h) {
    const StreamLayout& ly = plan.layout[(layer * a.n_kv + h) * 2 + 1];
    ntp = std::max(ntp, (ly.n2 + ly.n1 + 7) / 8);
  }
  const int npw = (ntp + 8 / gh - 1) / (8 / gh);
  a.stages = 3;
  if (GroupDigitSmem(gh, a.ks_max, a.n_words, 3).total > 227 * 1024) a.stages = 2;
  const size_t smem = static_cast<size_t>(GroupDigitSmem(gh, a.ks_max, a.n_words, a.stages).total);
  if (a.nq > 16 || npw > 24 || smem > 227 * 1024) return cudaErrorNotSupported;
  aatc_group_query_kernel<<<dim3(16, a.n_groups * gh, batch), kGQThreads, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 grid(a.n_splits, a.n_groups, batch);
  // pairs per warp: 12, 16 (g_h = 4 at ~2.75 bits: up to 32 value tiles per slice) or 24
  const void* kern = gh == 2 ? (npw <= 12 ? reinterpret_cast<const void*>(aatc_group_digit_kernel<2, 12>)
                                          : reinterpret_cast<const void*>(aatc_group_digit_kernel<2, 24>))
                             : (npw <= 12 ? reinterpret_cast<const void*>(aatc_group_digit_kernel<4, 12>)
                                : npw <= 16 ? reinterpret_cast<const void*>(aatc_group_digit_kernel<4, 16>)
                                            : reinterpret_cast<const void*>(aatc_group_digit_kernel<4, 24>));
  e = ensure_smem_optin(kern, smem);
  if (e != cudaSuccess) return e;
  if (gh == 2 && npw <= 12) aatc_group_digit_kernel<2, 12><<<grid, kGAThreads, smem, st>>>(a);
  else if (gh == 2) aatc_group_digit_kernel<2, 24><<<grid, kGAThreads, smem, st>>>(a);
  else if (npw <= 12) aatc_group_digit_kernel<4, 12><<<grid, kGAThreads, smem, st>>>(a);
  else if (npw <= 16) aatc_group_digit_kernel<4, 16><<<grid, kGAThreads, smem, st>>>(a);
  else aatc_group_digit_kernel<4, 24><<<grid, kGAThreads, smem, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t msm = static_cast<size_t>(a.n_splits) * 4;
  aatc_group_merge_kernel<<<dim3(a.nq, a.n_groups * gh, batch), kGMThreads, msm, st>>>(a);
  return cudaGetLastError();
}

}  // namespace aatc
