// AATC decode attention over the packed cache, the dequantization test hook, and the
// uncompressed bf16 reference decode (Def. sdpa with one query row; Algorithm 1
// "Reconstruct", "softmax", "Output" lines, computed without rebuilding the keys).
//
// Two launch plans, each a chain of programmatic dependents.  For layers whose key and value
// streams share one record shape (every per-stream plan at 1.5, 2, 2.75 or 4 bits) two launches
// per call: aatc_decode_fused_kernel (see there) rotates the queries and streams each split's
// tiles through per-warp-group rings, then the merge kernel below.  Any other layer takes three
// launches (flash-decoding split over the context):
//   query    per (sequence, kv-head, query slot): q' = (U_K^T q) f^K log2(e)/sqrt(128) for the
//            G query heads of the GQA group, the offset corrections C_g = sum_c q'_c 2^(b_c-1),
//            and q' per record entry as f16 hi/lo tensor-core fragments (mma.sync m16n8k16);
//   split    per (split, kv-head, sequence): pass 1 scores
//            s_{g,t} = alpha^K_t (sum_e q'_{g,e} digit_{t,e} - C_g) by f16 mma.sync over the
//            packed digits (each masked in place as a subnormal f16); split max m_g; pass 2
//            p = 2^(s - m_g), P' = p alpha^V_t as f16 hi/lo, value entry sums
//            sum_t P'_{g,t} digit_{t,e} by the same MMA; entry sums folded into channel sums with
//            the offset correction; (o, m, l) per split;
//   merge    per (sequence, query head): log-sum-exp merge of the splits, f^V / l, out = U_V o_hat.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <mutex>

#include "aatc_internal.h"
#include "ptx.cuh"

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
__device__ __forceinline__ void cp_async_wait_one() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

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

struct DecodeArgs {
  const uint32_t* words;   // cache word region (this layer)
  const float* alpha;      // cache alpha region
  const __nv_bfloat16* q;  // [batch][HQ][128]
  float* ws;               // [batch][HQ][n_splits][pstride]: o_c (128 channels), then m, l
  float* out;              // [batch][HQ][128]
  const float* u32;        // plan: [S][128 dim][128 ch]
  const float* u32t;       // plan: [S][128 ch][128 dim]
  const float* f;          // plan: [S][128]
  const ChanEnc* enc;      // plan: [S][128] (offsets 2^(b-1))
  const StreamLayout* lay; // plan: [S]
  const short* entry;      // plan: [S][n_entries]
  const short* chan_ent;   // plan: [S][128][kChanEnt] record entries of each channel (-1 padded)
  int* err;
  uint4* qfrag;            // workspace: score A fragments [batch][n_kv][ks_stride]
  float* qcorr;            // workspace: [batch][n_kv][16]: offset corrections C_g, score scales
  int layer, n_kv, n_q, group, n_ctx, n_tiles, n_words, n_entries, n_splits, split_len, ks_stride, pstride;
  int num_sms, cta_per_sm;  // split-kernel work permutation (cta_per_sm = 0: identity)
  int t_first;              // first packed token attended (tokens [t_first, n_ctx) of the cache)
  const __nv_bfloat16* k_full;  // uncompressed tokens attended as well: [batch][full_cap][n_kv][128]
  const __nv_bfloat16* v_full;
  int n_full, full_cap;
  int n_stages;             // fused kernel: tile ring depth
};

// 2^x with the hardware approximation (relative error ~2^-22; -inf -> 0)
__device__ __forceinline__ float fast_exp2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ float pow2i(int e) { return __int_as_float((127 + e) << 23); }   // 2^e, |e| < 127

constexpr int kWarps = kThreads / 32;

// Tensor-core formulation: mma.sync m16n8k16 with f16 operands and f32 accumulation.
//  * A packed 2-bit digit (or bit) masked into the low bits of a 16-bit half IS an f16 number:
//    the subnormal digit * 2^-24.  So an operand register (two digits) is one shift and one AND
//    of a record word, with no conversion.  (The e4m3 form of the same idea needs fewer masks,
//    but mma.sync with fp8 operands costs about a dozen instructions per MMA on this GPU, the
//    f16 form one.)
//  * The other operand (folded query, or probability P' = p alpha^V) is an f16 hi/lo pair,
//    hi = f16(x), lo = f16(x - hi), ~22 bits: row g of A holds hi and row g + 8 lo of query g,
//    so lane (g, t) accumulates hi (c0, c1) and lo (c2, c3) of query g separately and a query's
//    value is c0 + c2.  Products and their f32 sums were checked on the hardware to be exact for
//    subnormal digits; the accumulator keeps ~22 bits relative to its own magnitude.
//   scores:  B = record digits of 8 tokens.  One D2 word is one k16-step: b0 = word >> 2t
//            (fields t, t + 8), b1 = word >> 2t + 8 (fields t + 4, t + 12); one D1 word is two
//            k16-steps s: b0 = word >> t + 8s (fields t + 8s, t + 8s + 16), b1 = word >> t + 4 + 8s.
//   values:  B = value digits of one record entry for tokens (0, 2) and (1, 3) of a token quad,
//            from the quad-interleaved value words; A = P' of the same tokens in that order.
__device__ __forceinline__ void mma_f16(float (&c)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}

// f16 hi/lo split of two values, packed as (hi(x), hi(y)) and (lo(x), lo(y)); returns hi + lo.
__device__ __forceinline__ float2 f16_split2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x, y);
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(x - hf.x, y - hf.y);
  const float2 lf = __half22float2(l);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
  return make_float2(hf.x + lf.x, hf.y + lf.y);
}

constexpr float kOpMax = 16384.0f;            // |A operand| scaled to <= 2^14 (f16 max 65504)
constexpr float kDigitScale = 16777216.0f;    // a digit's f16 value is digit * 2^-24

constexpr int kQThreads = 512;
constexpr int kMaxEntries = 64 * 32;   // 16 bits x 128 channels

// Per call, per (sequence, kv-head, query slot g < 8): folded query q'_c = (U_K^T q)_c f_c
// log2(e)/sqrt(128), its offset correction C = sum_c q'_c 2^(b_c-1), the score scale, and rows g
// (hi) and g + 8 (lo) of the score A fragments: q'_c 2^shift per record entry, scaled so the
// largest is 2^14.  Slots g >= G write zero rows.
__global__ void __launch_bounds__(kQThreads)
    aatc_decode_query_kernel(const DecodeArgs a) {
  __shared__ float qv[D];
  __shared__ float part[4][D];
  __shared__ float xq[D];
  __shared__ float red[2][D / 32];
  __shared__ float xe[kMaxEntries];
  const int head = blockIdx.x, b = blockIdx.y, slot = blockIdx.z, tid = threadIdx.x;
  const int G = a.group;
  const bool real = slot < G;
  const int sk = (a.layer * a.n_kv + head) * 2;
  // every global input is requested up front (one memory round trip)
  const int c = tid & (D - 1), qd = tid >> 7;
  const short* ent = a.entry + static_cast<size_t>(sk) * a.n_entries;
  const short ce0 = tid < a.n_entries ? ent[tid] : 0;
  const short ce1 = tid + kQThreads < a.n_entries ? ent[tid + kQThreads] : 0;
  const StreamLayout lk = a.lay[sk];
  float qraw = 0.0f, fk = 0.0f, off = 0.0f;
  if (tid < D) {
    fk = a.f[sk * D + c];
    off = a.enc[sk * D + c].off;                                          // 2^(b_c - 1), 0 if b_c = 0
  }
  float u[32];
  {
    // thread (channel c, quarter qd of the dimensions)
    const float* uk = a.u32 + static_cast<size_t>(sk) * D * D + static_cast<size_t>(32 * qd) * D + c;
#pragma unroll
    for (int d = 0; d < 32; ++d) u[d] = uk[d * D];
  }
  // plan constants above; the query (and the workspace this call reuses) only once the preceding
  // grid in the stream is complete -- this kernel may be launched as its programmatic dependent
  ptx::grid_dependency_wait();
  // only now may the split kernel start: it reads the cache, which the preceding grid may write
  ptx::grid_launch_dependents();
  if (tid < D && real) qraw = __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + slot) * D + tid]);
  if (tid < D) qv[tid] = qraw;
  __syncthreads();
  {
    float acc = 0.0f;
#pragma unroll
    for (int d = 0; d < 32; ++d) acc = fmaf(u[d], qv[32 * qd + d], acc);
    part[qd][c] = acc;
  }
  __syncthreads();
  if (tid < D) {
    const float x = (part[0][c] + part[1][c] + part[2][c] + part[3][c]) * fk * (kLog2e * 0.08838834764831845f);
    float cr = x * off;
    float mx = fabsf(x) * off;                                             // largest |coefficient| of c
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      cr += __shfl_xor_sync(0xffffffffu, cr, o);
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if ((tid & 31) == 0) {
      red[0][tid >> 5] = cr;
      red[1][tid >> 5] = mx;
    }
    xq[c] = x;
  }
  __syncthreads();
  const float C = red[0][0] + red[0][1] + red[0][2] + red[0][3];
  const float m = fmaxf(fmaxf(red[1][0], red[1][1]), fmaxf(red[1][2], red[1][3]));
  const float inv = m > 0.0f ? kOpMax / m : 0.0f;                       // coefficients to |.| <= 2^14
  const int n_used = lk.n2 + lk.n1;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int e = tid + h * kQThreads;
    if (e < n_used) {
      const int ce = h ? ce1 : ce0;
      xe[e] = real ? xq[ce & 0xFF] * inv * pow2i(ce >> 8) : 0.0f;
    }
  }
  __syncthreads();
  // B fragments of the score MMA (tokens are the M rows, query columns the N = 8): head group
  // p = slot / 4 holds column g = slot % 4 (hi) and g + 4 (lo); lane (g, t) of k-step ks gets
  // (k 2t | 2t+1, k 2t+8 | 2t+9) of its column at fragment [ks][p][lane].
  const int n2w = lk.n2 / 16, n1w = (lk.n1 + 31) / 32;
  const int n_ks = n2w + 2 * n1w;
  const int np = (G + 3) / 4;
  if (slot >= 4 * np) return;                          // beyond the last head group
  const int p = slot >> 2, gs = slot & 3;
  uint2* dst = reinterpret_cast<uint2*>(a.qfrag + (static_cast<size_t>(b) * a.n_kv + head) * a.ks_stride);
  for (int i = tid; i < n_ks * 4; i += kQThreads) {
    const int ks = i >> 2, t = i & 3;
    int f[4];                                          // record fields of k = 2t, 2t+1, 2t+8, 2t+9
    int base, lim;
    if (ks < n2w) {
      f[0] = t; f[1] = t + 8; f[2] = t + 4; f[3] = t + 12;
      base = 16 * ks;
      lim = 16;
    } else {
      const int u = (ks - n2w) >> 1, sh = 8 * ((ks - n2w) & 1);
      f[0] = t + sh; f[1] = t + sh + 16; f[2] = t + 4 + sh; f[3] = t + 4 + sh + 16;
      base = lk.n2 + 32 * u;
      lim = min(32, lk.n1 - 32 * u);
    }
    float v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = f[k] < lim ? xe[base + f[k]] : 0.0f;
    // the split kernels mask digits in place: lane t's D2 digits arrive times 4^t, its D1 bits
    // times 2^t (k 2t, 2t+1) and 2^(t+4) (k 2t+8, 2t+9); the query rows carry the inverse.  (Only
    // bits 0..9 of a half are mantissa: the upper byte of each half is shifted down first, since
    // a digit in the exponent bits 10..15 would not be a multiple of the subnormal unit.)
    const float s01 = ks < n2w ? pow2i(-2 * t) : pow2i(-t);
    const float s89 = ks < n2w ? pow2i(-2 * t) : pow2i(-t - 4);
    v[0] *= s01;
    v[1] *= s01;
    v[2] *= s89;
    v[3] *= s89;
    uint32_t h01, l01, h89, l89;
    f16_split2(v[0], v[1], h01, l01);
    f16_split2(v[2], v[3], h89, l89);
    dst[(ks * np + p) * 32 + 4 * gs + t] = make_uint2(h01, h89);
    dst[(ks * np + p) * 32 + 4 * (gs + 4) + t] = make_uint2(l01, l89);
  }
  if (tid == 0) {
    float* qc = a.qcorr + (static_cast<size_t>(b) * a.n_kv + head) * 2 * MAX_GROUP;
    qc[slot] = real ? C : 0.0f;
    qc[MAX_GROUP + slot] = m > 0.0f ? m * (kDigitScale / kOpMax) : 0.0f;  // raw sum -> sum q' code
  }
}

constexpr int kStages = 3;                  // ring of record-word tiles (keys, then values)

__host__ __device__ constexpr int align16(int x) { return (x + 15) & ~15; }

// shared-memory carve-up of the split kernel (byte offsets)
struct SplitSmem {
  int bars, qcg, red, cetab, etab, afrag, ak, av, sbuf, pq, ring, total, sb_stride;
  __host__ __device__ SplitSmem(int n_ks, int np, int split_len, int W, int n_entries) {
    int o = 0;
    bars = o;  o = align16(o + 8 * (kStages + 1));  // ring barriers, then the prologue barrier
    qcg = o;   o += 2 * MAX_GROUP * 4;              // offset corrections, score scales
    red = o;   o += 4 * kWarps * MAX_GROUP * 4;     // reductions; per-query m, l, S', split max
    cetab = o; o += D * kChanEnt * 2;               // record entries of each value channel
    etab = o;  o = align16(o + n_entries * 2);      // value entry table (channel | shift << 8)
    afrag = o; o += n_ks * 32 * 16;                 // score A fragments per (k-step, lane)
    ak = o;    o += split_len * 4;                  // alpha^K, alpha^V of the split
    av = o;    o += split_len * 4;
    sb_stride = split_len + 8;                      // padded: query rows fall in different banks
    sbuf = o;  o += 4 * np * sb_stride * 4;         // scores of the split
    pq = o;    o += (TILE / 16) * 32 * 16;          // P' A fragments of one tile (8 k16-steps)
    ring = o;  o += kStages * W * TILE * 4;         // after the last tile: value entry sums
    total = o;
  }
};

// One CTA per (split, kv-head, sequence).  The split's record words stream through a ring of
// kStages tiles filled by bulk copies (keys of all its tiles, then values); alpha^K, alpha^V, the
// query fragments and the value entry tables arrive by bulk copy in the prologue.
// Pass 1: scores of the split; pass 2: P' and the value entry sums; then the entry sums become
// channel sums o_c = sum_e 2^shift O_e - 2^(b_c-1) S' (the Eq. 12 offset, folded after the
// product), written with the split's m and l for the merge kernel.
template <int JPW, int NP>
__global__ void __launch_bounds__(kThreads)
    aatc_decode_split_kernel(const DecodeArgs a) {
  extern __shared__ __align__(128) unsigned char smb[];
  __shared__ int s_abort;
  // Work item of this CTA.  CTAs i, i + S, i + 2S, ... (S SMs) tend to share an SM, and split
  // lengths follow a floor pattern with period S in that order, so without a permutation an SM
  // would get k splits of the same length; item = (i mod S) k + i / S gives every SM k
  // consecutive items instead (a near-equal share of tiles).
  int item = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);
  if (a.cta_per_sm > 0) item = (item % a.num_sms) * a.cta_per_sm + item / a.num_sms;
  const int split = item % a.n_splits, head = (item / a.n_splits) % a.n_kv, b = item / (a.n_splits * a.n_kv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;                       // mma fragment coordinates
  const int G = a.group;
  const int sk = (a.layer * a.n_kv + head) * 2, sv = sk + 1;   // key / value streams
  const StreamLayout lk = a.lay[sk], lv = a.lay[sv];
  const int W = a.n_words;
  const int n2w_k = lk.n2 / 16, n1w_k = (lk.n1 + 31) / 32;
  const int n_ks = n2w_k + 2 * n1w_k;                          // score k16-steps
  const int n2w_v = lv.n2 / 16, nw_v = n2w_v + (lv.n1 + 31) / 32;
  const SplitSmem L(n_ks, NP, a.split_len, W, a.n_entries);
  uint64_t* full = reinterpret_cast<uint64_t*>(smb + L.bars);
  uint64_t* pro = full + kStages;
  float* qcg = reinterpret_cast<float*>(smb + L.qcg);          // [0..7] C_g, [8..15] score scales
  float* red = reinterpret_cast<float*>(smb + L.red);
  const short* cetab = reinterpret_cast<const short*>(smb + L.cetab);
  const short* etab = reinterpret_cast<const short*>(smb + L.etab);
  const uint2* afrag = reinterpret_cast<const uint2*>(smb + L.afrag);  // [k-step][head group][lane]
  float* ak = reinterpret_cast<float*>(smb + L.ak);
  float* av = reinterpret_cast<float*>(smb + L.av);
  float* sbuf = reinterpret_cast<float*>(smb + L.sbuf);        // [4 NP][sb_stride]
  uint2* pq = reinterpret_cast<uint2*>(smb + L.pq);            // [8 k16-steps][head group][32 lanes]
  uint32_t* ring = reinterpret_cast<uint32_t*>(smb + L.ring);
  const int sbs = L.sb_stride;

  // tiles [tile_first, ceil(n_ctx / 128)) hold the attended packed tokens [t_first, n_ctx)
  const int tile_first = a.t_first / TILE;
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE - tile_first;
  const int tile_lo = tile_first + static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = tile_first + static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const int t_begin = tile_lo * TILE;                          // first token of the first tile
  const int t_lo = max(t_begin, a.t_first);                    // first attended token
  const int t_end = min(a.n_ctx, tile_hi * TILE);
  const int n_tiles_split = tile_hi - tile_lo;
  const int n_seq = 2 * n_tiles_split;                         // key tiles, then value tiles
  const int tile0 = tile_lo;
  const uint32_t tile_bytes = static_cast<uint32_t>(W) * TILE * 4;
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * W * TILE;
  const size_t bk = (static_cast<size_t>(b) * a.n_kv + head) * 2;   // cache stream of the keys
  const uint32_t* kwords = a.words + bk * stream_words;
  const uint32_t* vwords = a.words + (bk + 1) * stream_words;
  const float* kalpha = a.alpha + bk * a.n_tiles * TILE;
  const float* valpha = a.alpha + (bk + 1) * a.n_tiles * TILE;
  const float off_c = a.enc[sv * D + tid].off;                 // this thread's value channel
  ptx::grid_launch_dependents();                               // the merge kernel may get ready

  auto issue_tile = [&](int i) {
    const int s = i % kStages;
    const uint32_t* src = (i < n_tiles_split ? kwords : vwords) +
                          static_cast<size_t>(tile0 + i % n_tiles_split) * W * TILE;
    ptx::mbar_arrive_expect_tx(full + s, tile_bytes);
    ptx::bulk_load(ring + s * W * TILE, src, tile_bytes, full + s);
  };
  auto wait_tile = [&](int i) {
    if (!ptx::mbar_wait_sleep(full + i % kStages, (i / kStages) & 1, &s_abort, 32)) {
      s_abort = 1;
      atomicOr(a.err, 2);
    }
  };
  if (tid == 0) {
    s_abort = 0;
    for (int s2 = 0; s2 <= kStages; ++s2) ptx::mbar_init(full + s2, 1);
    ptx::fence_mbar_init();
    // cache words and scales do not depend on the query kernel: start them first
    const uint32_t abytes = static_cast<uint32_t>(n_tiles_split) * TILE * 4;
    const uint32_t ebytes = static_cast<uint32_t>(align16(a.n_entries * 2));
    const uint32_t fbytes = static_cast<uint32_t>(n_ks) * NP * 32 * 8;
    ptx::mbar_arrive_expect_tx(pro, 2 * abytes + D * kChanEnt * 2 + ebytes + fbytes + 2 * MAX_GROUP * 4);
    ptx::bulk_load(ak, kalpha + static_cast<size_t>(tile0) * TILE, abytes, pro);
    for (int i = 0; i < min(kStages, n_seq); ++i) issue_tile(i);
    ptx::bulk_load(av, valpha + static_cast<size_t>(tile0) * TILE, abytes, pro);
    ptx::bulk_load(smb + L.cetab, a.chan_ent + static_cast<size_t>(sv) * D * kChanEnt, D * kChanEnt * 2, pro);
    ptx::bulk_load(smb + L.etab, a.entry + static_cast<size_t>(sv) * a.n_entries, ebytes, pro);
    // the query kernel's fragments and corrections
    ptx::grid_dependency_wait();
    ptx::bulk_load(smb + L.afrag, a.qfrag + (static_cast<size_t>(b) * a.n_kv + head) * a.ks_stride, fbytes, pro);
    ptx::bulk_load(qcg, a.qcorr + (static_cast<size_t>(b) * a.n_kv + head) * 2 * MAX_GROUP, 2 * MAX_GROUP * 4, pro);
  }
  // P' columns of absent queries (q >= G) stay zero for the whole split
  for (int i = tid; i < (TILE / 16) * NP * 32; i += kThreads) {
    const int gcol = (i & 31) >> 2, q = 4 * ((i >> 5) % NP) + (gcol & 3);
    if (q >= G) pq[i] = make_uint2(0u, 0u);
  }
  __syncthreads();
  if (!ptx::mbar_wait_sleep(pro, 0, &s_abort, 200)) {
    s_abort = 1;
    atomicOr(a.err, 2);
  }

  // ---- pass 1: scores.  Warp = 32 tokens of each tile; lane (g, t) reads the record words of
  // tokens 4g .. 4g + 3 (one 128-bit load per k-step): M-tile 0 has rows g, g + 8 = tokens 4g,
  // 4g + 1, M-tile 1 tokens 4g + 2, 4g + 3; head group p gives the N = 8 query columns.
  const uint32_t m2 = 0x00030003u << (2 * t), m1a = 0x00010001u << t, m1b = 0x00010001u << (t + 4);
  // after the hi/lo exchange lane (g, t) owns heads 4p + 2(t & 1) + {0, 1} of tokens
  // 4g + 2 (t >> 1) + {0, 1}
  const int h_own = 2 * (t & 1), tk_own = 4 * g + 2 * (t >> 1);
  float mloc[NP][2];
  float sg[NP][2], cg[NP][2];
#pragma unroll
  for (int p = 0; p < NP; ++p)
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int q = 4 * p + h_own + i;
      mloc[p][i] = -INFINITY;
      sg[p][i] = q < G ? qcg[MAX_GROUP + q] : 0.0f;
      cg[p][i] = q < G ? qcg[q] : 0.0f;
    }
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    wait_tile(ti);
    const uint4* kt = reinterpret_cast<const uint4*>(ring + (ti % kStages) * W * TILE + 32 * warp + 4 * g);
    float acc[2][NP][4];
#pragma unroll
    for (int mh = 0; mh < 2; ++mh)
#pragma unroll
      for (int p = 0; p < NP; ++p)
#pragma unroll
        for (int r = 0; r < 4; ++r) acc[mh][p][r] = 0.0f;
    for (int ks = 0; ks < n2w_k; ++ks) {
      const uint4 x = kt[ks * (TILE / 4)];
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        const uint2 bf = afrag[(ks * NP + p) * 32 + lane];
        mma_f16(acc[0][p], make_uint4(x.x & m2, x.y & m2, (x.x >> 8) & m2, (x.y >> 8) & m2), bf.x, bf.y);
        mma_f16(acc[1][p], make_uint4(x.z & m2, x.w & m2, (x.z >> 8) & m2, (x.w >> 8) & m2), bf.x, bf.y);
      }
    }
    for (int u = 0; u < n1w_k; ++u) {
      const uint4 x = kt[(n2w_k + u) * (TILE / 4)];
#pragma unroll
      for (int hs = 0; hs < 2; ++hs) {
        const uint32_t y0 = hs ? x.x >> 8 : x.x, y1 = hs ? x.y >> 8 : x.y;
        const uint32_t y2 = hs ? x.z >> 8 : x.z, y3 = hs ? x.w >> 8 : x.w;
#pragma unroll
        for (int p = 0; p < NP; ++p) {
          const uint2 bf = afrag[((n2w_k + 2 * u + hs) * NP + p) * 32 + lane];
          mma_f16(acc[0][p], make_uint4(y0 & m1a, y1 & m1a, y0 & m1b, y1 & m1b), bf.x, bf.y);   // bits in place
          mma_f16(acc[1][p], make_uint4(y2 & m1a, y3 & m1a, y2 & m1b, y3 & m1b), bf.x, bf.y);
        }
      }
    }
    // columns 2t, 2t + 1 hold hi (t < 2) or lo (t >= 2) of heads 4p + 2(t & 1) + {0, 1}: lanes t
    // and t ^ 2 exchange so each owns the hi + lo sums of two tokens
    const int tk = ti * TILE + 32 * warp + tk_own;             // token of the split
    const float2 a2 = *reinterpret_cast<const float2*>(ak + tk);
    const int tb = t_begin + tk;
    const bool ok0 = tb >= t_lo && tb < t_end, ok1 = tb + 1 >= t_lo && tb + 1 < t_end;
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      float r[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float mine = t < 2 ? acc[0][p][i] : acc[1][p][i];
        const float give = t < 2 ? acc[1][p][i] : acc[0][p][i];
        r[i] = mine + __shfl_xor_sync(0xffffffffu, give, 2);
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int q = 4 * p + h_own + i;
        if (q < G) {
          const float s0 = ok0 ? a2.x * fmaf(r[i], sg[p][i], -cg[p][i]) : -INFINITY;       // c0 / c1: token A
          const float s1 = ok1 ? a2.y * fmaf(r[2 + i], sg[p][i], -cg[p][i]) : -INFINITY;   // c2 / c3: token B
          *reinterpret_cast<float2*>(sbuf + q * sbs + tk) = make_float2(s0, s1);
          mloc[p][i] = fmaxf(mloc[p][i], fmaxf(s0, s1));
        }
      }
    }
    __syncthreads();                                           // stage free: refill
    if (tid == 0 && ti + kStages < n_seq) {
      ptx::fence_proxy_async_smem();
      issue_tile(ti + kStages);
    }
  }
  // split max per query; largest alpha^V of the split (P' = p alpha^V is coded relative to it)
  float amx = 0.0f;
  for (int i = t_lo - t_begin + tid; i < t_end - t_begin; i += kThreads) amx = fmaxf(amx, av[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amx = fmaxf(amx, __shfl_xor_sync(0xffffffffu, amx, o));
  if (lane == 0) red[3 * kWarps * MAX_GROUP + warp] = amx;
#pragma unroll
  for (int p = 0; p < NP; ++p)
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      float v = mloc[p][i];
      v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
      v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
      v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
      v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
      if (lane < 2) red[warp * MAX_GROUP + 4 * p + 2 * lane + i] = v;      // lane t = lane < 2
    }
  __syncthreads();
  float* mqs = red + 2 * kWarps * MAX_GROUP + 3 * MAX_GROUP;  // [MAX_GROUP] split max per query
  if (tid < MAX_GROUP)
    mqs[tid] = fmaxf(fmaxf(red[0 * MAX_GROUP + tid], red[1 * MAX_GROUP + tid]),
                     fmaxf(red[2 * MAX_GROUP + tid], red[3 * MAX_GROUP + tid]));
  {
    const float* am = red + 3 * kWarps * MAX_GROUP;
    amx = fmaxf(fmaxf(am[0], am[1]), fmaxf(am[2], am[3]));
  }
  const float inv_p = amx > 0.0f ? kOpMax / amx : 0.0f;       // P' to |.| <= 2^14
  const float val_scale = amx * (kDigitScale / kOpMax);        // raw sum -> sum P' code
  __syncthreads();                                             // split maxima visible to pass 2

  // ---- pass 2: P' (thread = 4 tokens x 1 query) and the value product over the split.
  // Value M-tiles ("jobs", 16 record entries each): a D2 word is one (fields g, g + 8 of lane row
  // g: slots 2(g / 4), 2(g / 4) + 1 of a token quad), a D1 word two (quarters 0, 1 or 2, 3:
  // slots hb, hb + 2).  Lane (g, t) of k-step ks reads token quad 4 ks + t; per job it keeps the
  // offsets of its two slots in the tile and its field mask.  Warp w takes jobs
  // [w J / 4, (w+1) J / 4).
  const int n_jobs = n2w_v + 2 * (nw_v - n2w_v);
  const int j0 = warp * n_jobs / kWarps, nj = (warp + 1) * n_jobs / kWarps - j0;
  int joff[JPW], jsec[JPW];
  uint32_t jmask[JPW];
#pragma unroll
  for (int j = 0; j < JPW; ++j) {
    const int jj = j0 + j;
    // fields masked in place: a row gets digit * 4^(g & 3) (D2) or bit * 2^g (D1), divided out
    // of the entry sums in the epilogue
    if (jj < n2w_v) {
      joff[j] = jj * TILE + 2 * (g >> 2);
      jsec[j] = 1;
      jmask[j] = 0x00030003u << (2 * (g & 3));
    } else {
      const int u = jj - n2w_v;
      joff[j] = (n2w_v + (u >> 1)) * TILE + (u & 1);
      jsec[j] = 2;
      jmask[j] = 0x00010001u << g;
    }
  }
  float vacc[JPW][NP][4];
#pragma unroll
  for (int j = 0; j < JPW; ++j)
#pragma unroll
    for (int p = 0; p < NP; ++p)
#pragma unroll
      for (int z = 0; z < 4; ++z) vacc[j][p][z] = 0.0f;
  float lsum[NP], ssum[NP];
#pragma unroll
  for (int p = 0; p < NP; ++p) lsum[p] = ssum[p] = 0.0f;
  {
    // tokens 4 Q .. 4 Q + 3 with Q = 8 warp + Qk (k-step Q / 4, fragment lane column t = Q % 4)
    const int qq = lane >> 3, Qk = lane & 7, Q = 8 * warp + Qk;
    const int tk0 = 4 * Q;
    for (int ti = 0; ti < n_tiles_split; ++ti) {
      const int i_seq = n_tiles_split + ti;
      wait_tile(i_seq);
      const uint32_t* vt = ring + (i_seq % kStages) * W * TILE;
      {
        const int tq = (tile0 + ti) * TILE + tk0;                // first token of this quad
        const float4 a4 = *reinterpret_cast<const float4*>(av + ti * TILE + tk0);
        const float av0 = tq >= t_lo && tq < t_end ? a4.x * inv_p : 0.0f;
        const float av1 = tq + 1 >= t_lo && tq + 1 < t_end ? a4.y * inv_p : 0.0f;
        const float av2 = tq + 2 >= t_lo && tq + 2 < t_end ? a4.z * inv_p : 0.0f;
        const float av3 = tq + 3 >= t_lo && tq + 3 < t_end ? a4.w * inv_p : 0.0f;
#pragma unroll
        for (int p = 0; p < NP; ++p) {
          const int q = 4 * p + qq;
          if (q < G) {
            const float4 sc = *reinterpret_cast<const float4*>(sbuf + q * sbs + ti * TILE + tk0);
            const float mq = mqs[q];
            const float p0 = fast_exp2(sc.x - mq), p1 = fast_exp2(sc.y - mq);
            const float p2 = fast_exp2(sc.z - mq), p3 = fast_exp2(sc.w - mq);
            lsum[p] += (p0 + p1) + (p2 + p3);
            uint32_t h02, l02, h13, l13;
            const float2 r02 = f16_split2(p0 * av0, p2 * av2, h02, l02);   // tokens 0, 2 (k 2t, 2t+1)
            const float2 r13 = f16_split2(p1 * av1, p3 * av3, h13, l13);   // tokens 1, 3 (k 2t+8, 2t+9)
            ssum[p] += (r02.x + r02.y) + (r13.x + r13.y);                  // what the MMA sees
            uint2* dst = pq + ((Q >> 2) * NP + p) * 32 + (Q & 3);
            dst[4 * qq] = make_uint2(h02, h13);                            // column qq: hi
            dst[4 * (qq + 4)] = make_uint2(l02, l13);                      // column qq + 4: lo
          }
        }
      }
      __syncthreads();
#pragma unroll
      for (int ks = 0; ks < TILE / 16; ++ks) {
        uint2 bf[NP];
#pragma unroll
        for (int p = 0; p < NP; ++p) bf[p] = pq[(ks * NP + p) * 32 + lane];   // column g, quad 4 ks + t
#pragma unroll
        for (int j = 0; j < JPW; ++j)
          if (j < nj) {
            const uint32_t* src = vt + joff[j] + 4 * (4 * ks + t);
            const uint32_t xa = src[0], xb = src[jsec[j]];
            const uint32_t mk = jmask[j];
            const uint4 af = make_uint4(xa & mk, xb & mk, (xa >> 8) & mk, (xb >> 8) & mk);
#pragma unroll
            for (int p = 0; p < NP; ++p) mma_f16(vacc[j][p], af, bf[p].x, bf[p].y);
          }
      }
      __syncthreads();                                         // stage and pq free: refill
      if (tid == 0 && i_seq + kStages < n_seq) {
        ptx::fence_proxy_async_smem();
        issue_tile(i_seq + kStages);
      }
    }
  }

  // ---- per-query m, l, S' of the split; value entry sums into shared memory (drained ring)
#pragma unroll
  for (int p = 0; p < NP; ++p)
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      lsum[p] += __shfl_xor_sync(0xffffffffu, lsum[p], o);
      ssum[p] += __shfl_xor_sync(0xffffffffu, ssum[p], o);
    }
  float* oe = reinterpret_cast<float*>(ring);                  // [G][n_entries]: the ring is drained
  if ((lane & 7) == 0)
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      red[warp * MAX_GROUP + 4 * p + (lane >> 3)] = lsum[p];
      red[(kWarps + warp) * MAX_GROUP + 4 * p + (lane >> 3)] = ssum[p];
    }
  {
    // columns 2t, 2t + 1: hi (t < 2) / lo (t >= 2) of heads 4p + 2(t & 1) + {0, 1}; after the
    // exchange lanes t < 2 own entry row g, lanes t >= 2 entry row g + 8
#pragma unroll
    for (int j = 0; j < JPW; ++j) {
      const int jj = j0 + j;
      int e = 0;
      float sc = 0.0f;
      if (jj < n2w_v) {
        e = 16 * jj + g + 8 * (t >> 1);
        sc = val_scale * pow2i(-2 * (g & 3));
      } else {
        const int u = jj - n2w_v;
        e = lv.n2 + 32 * (u >> 1) + 16 * (u & 1) + g + 8 * (t >> 1);
        sc = val_scale * pow2i(-g);
      }
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        float r[2];
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const float mine = t < 2 ? vacc[j][p][i] : vacc[j][p][2 + i];
          const float give = t < 2 ? vacc[j][p][2 + i] : vacc[j][p][i];
          r[i] = mine + __shfl_xor_sync(0xffffffffu, give, 2);
        }
        if (j < nj && e < lv.n2 + lv.n1)
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            const int q = 4 * p + h_own + i;
            if (q < G) oe[q * a.n_entries + e] = r[i] * sc;
          }
      }
    }
  }
  __syncthreads();
  float* ml = red + 2 * kWarps * MAX_GROUP;                    // [3][MAX_GROUP]: m, l, S'
  if (tid < G) {
    const int q = tid;
    ml[q] = mqs[q];
    ml[MAX_GROUP + q] = red[q] + red[MAX_GROUP + q] + red[2 * MAX_GROUP + q] + red[3 * MAX_GROUP + q];
    ml[2 * MAX_GROUP + q] = (red[(kWarps + 0) * MAX_GROUP + q] + red[(kWarps + 1) * MAX_GROUP + q] +
                             red[(kWarps + 2) * MAX_GROUP + q] + red[(kWarps + 3) * MAX_GROUP + q]) *
                            (amx / kOpMax);
  }
  __syncthreads();
  // channel sums of this split: thread = channel
  const size_t pbase = (static_cast<size_t>(b) * a.n_q + head * G) * a.n_splits;
  {
    const int c = tid;
    // up to kChanEnt record entries of the channel (more than 8 only for widths above 8)
    const short* ce = cetab + c * kChanEnt;
    const int nce = ce[8] >= 0 ? kChanEnt : 8;
    float w[kChanEnt];
    int e_[kChanEnt];
#pragma unroll
    for (int k = 0; k < kChanEnt; ++k) {
      const int ek = k < nce ? ce[k] : -1;
      e_[k] = min(max(ek, 0), a.n_entries - 1);
      w[k] = ek >= 0 ? pow2i((etab[e_[k]] >> 8) & 15) : 0.0f;
    }
    const float off = off_c;
    for (int q = 0; q < G; ++q) {
      float o = -off * ml[2 * MAX_GROUP + q];
#pragma unroll
      for (int k = 0; k < kChanEnt; ++k) o = fmaf(w[k], oe[q * a.n_entries + e_[k]], o);
      float* dst = a.ws + (pbase + static_cast<size_t>(q) * a.n_splits + split) * a.pstride;
      dst[c] = o;
      if (c == 0) {
        dst[D] = ml[q];
        dst[D + 1] = ml[MAX_GROUP + q];
      }
    }
  }
}

// ---------------------------------------------------------------- fused split + merge kernel
// For plans whose key and value streams of the layer share one record shape (N2W D2 words, N1W D1
// words).  CTA = (split, kv-head, sequence) with WG warp groups of four warps, one CTA per SM in
// one wave; the query rotation is folded in (every CTA rotates its group's queries itself, while
// its first tiles are in flight) and the split's partial (o, m, l) per query goes to the
// workspace for the merge kernel, which follows as this grid's programmatic dependent.  (A merge
// by the last CTA of each (sequence, kv-head), behind completion flags, measured slower: its
// fences, flag round and serial partial reads cost more than the grid boundary.)
//  * Warp group wg takes tiles wg, wg + WG, ... of the split through its own ring of NS stages (a
//    tile's keys, values and scales arrive together in one stage; the last of the group's four
//    warps to finish a stage refills it).  Each warp owns a quarter (32 tokens) of a tile and runs
//    its own online softmax, keys then values of the same tile, so warps never wait for each
//    other inside the loop.
//  * Reference maximum m per query, kept within 2^8 of the running maximum of e_t = s_t +
//    floor(log2 alpha^V_t) (floored at s_t - 64), and raised (with the sums rescaled) only when a
//    tile exceeds it by more than that: the value weight P' = 2^(s - m) alpha^V stays below 2^9
//    and p = 2^(s - m) below 2^72 whatever the scales, so the split needs no pass over its alpha
//    values first.  m is only a reference point: o = sum P' code and l = sum p share it, and the
//    merge rescales both alike.
__host__ __device__ constexpr int fused_stage_bytes(int wu) { return 2 * wu * TILE * 4 + 2 * TILE * 4; }
// row pitch of the per-query entry sums in the epilogue: = 8 (mod 16), so the four queries of a
// lane quad (rows t = 0..3) fall in distinct banks
__host__ __device__ constexpr int fused_entry_pitch(int n_entries) { return ((n_entries + 7) / 8 * 8) | 8; }
constexpr float kPScale = 32.0f;            // P' < 2^9 times 2^5: f16 operands below 2^14

struct FusedSmem {
  int bars, cnt, qf, qc, pf, cetab, cw8, ketab, fold, ring, total;
  __host__ __device__ FusedSmem(int wu, int nks, int np, int wg, int n_entries, int n_stages) {
    const int gmax = 4 * np, warps = 4 * wg;
    int o = 0;
    bars = o;  o = align16(o + 8 * wg * n_stages);
    cnt = o;   o = align16(o + 4 * wg * n_stages);
    qf = o;    o += nks * np * 32 * 8;                        // query B fragments [ks][p][lane]
    qc = o;    o += 2 * MAX_GROUP * 4 + D * 4;                // C_g, score scales; value offsets 2^(b_c - 1)
    pf = o;    o += warps * 2 * np * 32 * 8;                  // P' B fragments [warp][ks][p][lane]
    cetab = o; o += D * 8 * 2;                                // value channel -> its record entries (clamped)
    cw8 = o;   o += D * 8 * 4;                                // 2^shift of those entries (0: none)
    ketab = o; o = align16(o + n_entries * 2);                // key entry table
    fold = o;  o += ((2 + wg) * gmax * D + 2 * warps * gmax) * 4;   // q, q', partial q' [wg]; reductions
    o = (o + 127) & ~127;
    ring = o;
    const int rings = wg * n_stages * fused_stage_bytes(wu);
    // after the loop the rings hold each warp's (m, l, S', entry sums) per query, the warps'
    // factors 2^(m_w - M), the totals (M, l, S') and the entry sums over the warps
    const int nep = fused_entry_pitch(n_entries);
    const int epi = (warps * (3 * MAX_GROUP + gmax * nep) + warps * gmax + 3 * gmax + gmax * nep) * 4;
    total = ring + (rings > epi ? rings : epi);
  }
};

template <int N2W, int N1W, int NP, int WG>
__global__ void __launch_bounds__(128 * WG, 1)
    aatc_decode_fused_kernel(const DecodeArgs a) {
  constexpr int WU = N2W + N1W;                  // record words the streams use
  constexpr int NKS = N2W + 2 * N1W;             // score k16-steps
  constexpr int NJ = N2W + 2 * N1W;              // value M-tiles (16 record entries each)
  constexpr int GMAX = 4 * NP;
  constexpr int NW = 4 * WG;                     // warps
  constexpr int NT = 32 * NW;                    // threads
  constexpr uint32_t kTileWords = WU * TILE;
  constexpr uint32_t kStage = fused_stage_bytes(WU);
  extern __shared__ __align__(128) unsigned char smb[];
  __shared__ int s_abort, s_never, s_issued[WG];
  int item = blockIdx.x;
  if (a.cta_per_sm > 0) item = (item % a.num_sms) * a.cta_per_sm + item / a.num_sms;
  const int split = item % a.n_splits, head = (item / a.n_splits) % a.n_kv, b = item / (a.n_splits * a.n_kv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wg = warp >> 2, wq = warp & 3;       // warp group, token quarter
  const int g = lane >> 2, t = lane & 3;
  const int G = a.group;
  const int NS = a.n_stages;
  const int sk = (a.layer * a.n_kv + head) * 2, sv = sk + 1;
  const FusedSmem L(WU, NKS, NP, WG, a.n_entries, NS);
  uint64_t* full = reinterpret_cast<uint64_t*>(smb + L.bars) + wg * NS;   // this group's ring barriers
  int* cnt = reinterpret_cast<int*>(smb + L.cnt) + wg * NS;
  const uint2* qf = reinterpret_cast<const uint2*>(smb + L.qf);
  unsigned char* pfw = smb + L.pf + warp * (2 * NP * 32 * 8);
  const short* cetab = reinterpret_cast<const short*>(smb + L.cetab);
  const float* cw8 = reinterpret_cast<const float*>(smb + L.cw8);
  const short* ketab = reinterpret_cast<const short*>(smb + L.ketab);
  unsigned char* ring = smb + L.ring + wg * NS * kStage;

  const int tile_first = a.t_first / TILE;
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE - tile_first;
  const int tile_lo = tile_first + static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = tile_first + static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const int t_lo = a.t_first, t_end = a.n_ctx;
  const int n_tl = tile_hi - tile_lo;
  const int n_j = n_tl > wg ? (n_tl - wg + WG - 1) / WG : 0;     // tiles of this warp group
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;
  const size_t bk = (static_cast<size_t>(b) * a.n_kv + head) * 2;
  const uint32_t* kwords = a.words + bk * stream_words;
  const uint32_t* vwords = kwords + stream_words;
  const float* kalpha = a.alpha + bk * a.n_tiles * TILE;
  const float* valpha = kalpha + static_cast<size_t>(a.n_tiles) * TILE;

  auto issue = [&](int j, int s) {             // the group's j-th tile into stage s = j mod NS
    unsigned char* st = ring + s * kStage;
    const int tile = tile_lo + wg + WG * j;
    const size_t tw = static_cast<size_t>(tile) * a.n_words * TILE;
    const size_t ta = static_cast<size_t>(tile) * TILE;
    // the cache is read once per call: evict-first keeps the plan tables in L2
    const uint64_t pol = ptx::l2_policy_evict_first();
    ptx::mbar_arrive_expect_tx(full + s, kStage);
    ptx::bulk_load_hint(st, kwords + tw, kTileWords * 4, full + s, pol);
    ptx::bulk_load_hint(st + kTileWords * 4, vwords + tw, kTileWords * 4, full + s, pol);
    ptx::bulk_load_hint(st + 2 * kTileWords * 4, kalpha + ta, TILE * 4, full + s, pol);
    ptx::bulk_load_hint(st + 2 * kTileWords * 4 + TILE * 4, valpha + ta, TILE * 4, full + s, pol);
    s_issued[wg] = j + 1;
  };
  const bool leader = (tid & 127) == 0;          // thread 0 of a warp group
  if (leader) {
    s_issued[wg] = 0;
    for (int s = 0; s < NS; ++s) ptx::mbar_init(full + s, 1);
    ptx::fence_mbar_init();
  }
  if (tid == 0) {
    s_abort = 0;
    s_never = 0;
  }
  // plan constants (never written by a kernel): the streams' entry tables, key channel constants
  // (the first 8 entries of each channel: all of them for widths up to 8, the only plans this
  // kernel is launched for)
  for (int i = tid; i < D * 8; i += NT) {
    const int ce = a.chan_ent[(static_cast<size_t>(sv) * D + (i >> 3)) * kChanEnt + (i & 7)];
    const int e = min(max(ce, 0), a.n_entries - 1);
    reinterpret_cast<short*>(smb + L.cetab)[i] = static_cast<short>(e);
    reinterpret_cast<float*>(smb + L.cw8)[i] =
        ce >= 0 ? pow2i((a.entry[static_cast<size_t>(sv) * a.n_entries + e] >> 8) & 15) : 0.0f;
  }
  for (int i = tid; i < a.n_entries; i += NT)
    reinterpret_cast<short*>(smb + L.ketab)[i] = a.entry[static_cast<size_t>(sk) * a.n_entries + i];
  const int c = tid & (D - 1), part = tid >> 7;                 // channel, part of the fold (WG parts)
  // U_K rows of this thread's part of the fold: plan constants, requested before the wait
  constexpr int DR = D / WG, RR = DR < 64 ? DR : 64;
  const float* uk = a.u32 + static_cast<size_t>(sk) * D * D + static_cast<size_t>(part * DR) * D + c;
  float u0[RR];
#pragma unroll
  for (int k = 0; k < RR; ++k) u0[k] = __ldg(uk + k * D);
  const float fk = a.f[sk * D + c];
  const float offk = a.enc[sk * D + c].off;                     // 2^(b_c - 1), 0 if b_c = 0
  if (tid < D) reinterpret_cast<float*>(smb + L.qc)[2 * MAX_GROUP + tid] = a.enc[sv * D + tid].off;
  const StreamLayout lk = a.lay[sk];
  if (tid < WG * NS) reinterpret_cast<int*>(smb + L.cnt)[tid] = 0;
  // everything below may read what the preceding grid in the stream wrote (cache, q, workspace)
  ptx::grid_dependency_wait();
  if (leader && n_j > 0) issue(0, 0);          // first tile now, the rest of the ring after the fold

  // ---- query rotation and fold, while the first tiles are in flight:
  //   q'_{g,c} = (U_K^T q_g)_c f^K_c log2(e) / sqrt(128),  C_g = sum_c q'_{g,c} 2^(b_c - 1),
  // and the score B fragments: q'_{g,c(e)} 2^shift(e) per record entry e, scaled so the largest
  // is 2^14, as f16 hi / lo; columns 2 gs (hi) and 2 gs + 1 (lo) of query group p for query 4p + gs
  float* qv = reinterpret_cast<float*>(smb + L.fold);           // [GMAX][128] q
  float* xq = qv + GMAX * D;                                    // [GMAX][128] q'
  float* xpart = xq + GMAX * D;                                 // [WG][GMAX][128] partial U_K^T q
  float* fred = xpart + WG * GMAX * D;                          // [2][NW][GMAX]
  for (int i = tid; i < GMAX * D; i += NT) {
    const int gq = i >> 7;
    qv[i] = gq < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + gq) * D + (i & (D - 1))]) : 0.0f;
  }
  __syncthreads();
  {
    // part p of the thread sums dimensions [p D / WG, (p + 1) D / WG), RR rows of U_K in flight
    float acc[GMAX];
#pragma unroll
    for (int q = 0; q < GMAX; ++q) acc[q] = 0.0f;
#pragma unroll 1
    for (int r = 0; r < DR / RR; ++r) {
      float u[RR];
#pragma unroll
      for (int k = 0; k < RR; ++k) u[k] = r == 0 ? u0[k] : __ldg(uk + (RR * r + k) * D);
#pragma unroll
      for (int k4 = 0; k4 < RR / 4; ++k4)
#pragma unroll
        for (int q = 0; q < GMAX; ++q) {
          const float4 qq = *reinterpret_cast<const float4*>(qv + q * D + part * DR + RR * r + 4 * k4);
          acc[q] = fmaf(u[4 * k4], qq.x, acc[q]);
          acc[q] = fmaf(u[4 * k4 + 1], qq.y, acc[q]);
          acc[q] = fmaf(u[4 * k4 + 2], qq.z, acc[q]);
          acc[q] = fmaf(u[4 * k4 + 3], qq.w, acc[q]);
        }
    }
#pragma unroll
    for (int q = 0; q < GMAX; ++q) xpart[(part * GMAX + q) * D + c] = acc[q];
  }
  __syncthreads();
  if (part == 0) {
#pragma unroll
    for (int q = 0; q < GMAX; ++q) {
      float sum = 0.0f;
#pragma unroll
      for (int p2 = 0; p2 < WG; ++p2) sum += xpart[(p2 * GMAX + q) * D + c];
      const float x = sum * fk * (kLog2e * 0.08838834764831845f);
      xq[q * D + c] = x;
      float cr = x * offk, mx = fabsf(x) * offk;                  // largest |coefficient| of c
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        cr += __shfl_xor_sync(0xffffffffu, cr, o);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      }
      if (lane == 0) {
        fred[warp * GMAX + q] = cr;
        fred[(NW + warp) * GMAX + q] = mx;
      }
    }
  }
  __syncthreads();
  {
    float* qcw = reinterpret_cast<float*>(smb + L.qc);
    if (tid < GMAX) {
      const int q = tid;
      float cs = 0.0f, m = 0.0f;
#pragma unroll
      for (int w = 0; w < 4; ++w) {                               // the four warps of part 0
        cs += fred[w * GMAX + q];
        m = fmaxf(m, fred[(NW + w) * GMAX + q]);
      }
      qcw[q] = q < G ? cs : 0.0f;
      qcw[MAX_GROUP + q] = q < G && m > 0.0f ? m * (kDigitScale / kOpMax) : 0.0f;   // raw sum -> sum q' u
    }
    // lane t of k-step ks holds fields (k 2t, 2t+1, 2t+8, 2t+9) = D2 (t, t+8, t+4, t+12) of word
    // ks, or D1 bits (t, t+16, t+4, t+20) + 8 hs of word u for k-step ks = N2W + 2u + hs; the
    // split loop masks them in place (times 4^t, or 2^t and 2^(t+4)), the fragments divide it out
    uint2* qfw = reinterpret_cast<uint2*>(smb + L.qf);
    for (int i = tid; i < NKS * 4 * GMAX; i += NT) {
      const int q = i % GMAX, tt = (i / GMAX) & 3, ks = i / (4 * GMAX);
      float mq = 0.0f;                                            // largest |coefficient| of query q
#pragma unroll
      for (int w = 0; w < 4; ++w) mq = fmaxf(mq, fred[(NW + w) * GMAX + q]);
      const float invq = mq > 0.0f ? kOpMax / mq : 0.0f;
      int f[4], base, lim;
      float s01, s89;
      if (ks < N2W) {
        f[0] = tt; f[1] = tt + 8; f[2] = tt + 4; f[3] = tt + 12;
        base = 16 * ks;
        lim = 16;
        s01 = s89 = pow2i(-2 * tt);
      } else {
        const int u = (ks - N2W) >> 1, sh = 8 * ((ks - N2W) & 1);
        f[0] = tt + sh; f[1] = tt + sh + 16; f[2] = tt + 4 + sh; f[3] = tt + 4 + sh + 16;
        base = lk.n2 + 32 * u;
        lim = min(32, lk.n1 - 32 * u);
        s01 = pow2i(-tt);
        s89 = pow2i(-tt - 4);
      }
      float v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int ce = f[k] < lim && q < G ? ketab[base + f[k]] : 0;
        v[k] = f[k] < lim && q < G ? xq[q * D + (ce & 0xFF)] * invq * pow2i(ce >> 8) * (k < 2 ? s01 : s89) : 0.0f;
      }
      uint32_t h01, l01, h89, l89;
      f16_split2(v[0], v[1], h01, l01);
      f16_split2(v[2], v[3], h89, l89);
      const int p = q >> 2, gs = q & 3;
      qfw[(ks * NP + p) * 32 + 4 * (2 * gs) + tt] = make_uint2(h01, h89);        // column 2 gs: hi
      qfw[(ks * NP + p) * 32 + 4 * (2 * gs + 1) + tt] = make_uint2(l01, l89);    // column 2 gs + 1: lo
    }
  }
  const float* qc = reinterpret_cast<const float*>(smb + L.qc);
  ptx::grid_launch_dependents();
  __syncthreads();
  // the rest of each group's ring: lane 0 of the group's last warp, which starts its first tile
  // after the other three (they need only the tile issued before the fold)
  if ((tid & 127) == 96)
    for (int j = 1; j < min(NS, n_j); ++j) issue(j, j);

  // masks: scores (lane t's fields of a k-step), values (lane row g's fields of an M-tile)
  const uint32_t km2 = 0x00030003u << (2 * t);
  const uint32_t km1a = 0x00010001u << t, km1b = 0x00010001u << (t + 4);
  const uint32_t vm2 = 0x00030003u << (2 * (g & 3));
  const uint32_t vm1 = 0x00010001u << g;
  const int d2off = 2 * (g >> 2);
  // With the hi and lo columns of a query side by side, lane (g, t)'s accumulators c0 + c1 and
  // c2 + c3 are whole sums for query 4p + t: in the key pass of tokens 4g + {0, 1} (M-tile 0) and
  // 4g + {2, 3} (M-tile 1), i.e. the lane owns query 4p + t over the token quad g of its warp; in
  // the value pass of record-entry rows g and g + 8
  const int tq = 32 * wq + 4 * g;                // first token of the lane's quad in a tile
  float sg[NP], cg[NP], mrun[NP], lsum[NP], ssum[NP];
#pragma unroll
  for (int p = 0; p < NP; ++p) {
    const int q = 4 * p + t;
    sg[p] = q < G ? qc[MAX_GROUP + q] : 0.0f;
    cg[p] = q < G ? qc[q] : 0.0f;
    mrun[p] = -INFINITY;
    lsum[p] = 0.0f;
    ssum[p] = 0.0f;
  }
  float vacc[NJ][NP][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j)
#pragma unroll
    for (int p = 0; p < NP; ++p)
#pragma unroll
      for (int z = 0; z < 4; ++z) vacc[j][p][z] = 0.0f;

  int s = 0;                                     // stage of tile j and the parity of its phase
  uint32_t ph = 0;
  for (int j = 0; j < n_j; ++j) {
    if (!ptx::mbar_wait_sleep(full + s, ph, &s_abort, 20)) {
      s_abort = 1;
      atomicOr(a.err, 2);
    }
    if (s_abort) break;
    const int ti = wg + WG * j;                  // tile of the split
    const unsigned char* st = ring + s * kStage;
    const uint32_t* kt = reinterpret_cast<const uint32_t*>(st);
    const uint32_t* vt = kt + kTileWords;
    const float* ak = reinterpret_cast<const float*>(vt + kTileWords);
    const float* av = ak + TILE;
    // ---- scores of the warp's 32 tokens: M-tile 0 rows (g, g + 8) = tokens 4g, 4g + 1, M-tile 1
    // tokens 4g + 2, 4g + 3; N = 8 columns of query group p (hi, lo of queries 4p .. 4p + 3)
    float kacc[2][NP][4];
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
      for (int p = 0; p < NP; ++p)
#pragma unroll
        for (int z = 0; z < 4; ++z) kacc[m][p][z] = 0.0f;
    const uint4* kp = reinterpret_cast<const uint4*>(kt + tq);
#pragma unroll
    for (int ks = 0; ks < N2W; ++ks) {
      const uint4 x = kp[ks * (TILE / 4)];
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        const uint2 bf = qf[(ks * NP + p) * 32 + lane];
        mma_f16(kacc[0][p], make_uint4(x.x & km2, x.y & km2, (x.x >> 8) & km2, (x.y >> 8) & km2), bf.x, bf.y);
        mma_f16(kacc[1][p], make_uint4(x.z & km2, x.w & km2, (x.z >> 8) & km2, (x.w >> 8) & km2), bf.x, bf.y);
      }
    }
#pragma unroll
    for (int u = 0; u < N1W; ++u) {
      const uint4 x = kp[(N2W + u) * (TILE / 4)];
#pragma unroll
      for (int hs = 0; hs < 2; ++hs) {
        const uint4 y = hs ? make_uint4(x.x >> 8, x.y >> 8, x.z >> 8, x.w >> 8) : x;
#pragma unroll
        for (int p = 0; p < NP; ++p) {
          const uint2 bf = qf[((N2W + 2 * u + hs) * NP + p) * 32 + lane];
          mma_f16(kacc[0][p], make_uint4(y.x & km1a, y.y & km1a, y.x & km1b, y.y & km1b), bf.x, bf.y);
          mma_f16(kacc[1][p], make_uint4(y.z & km1a, y.w & km1a, y.z & km1b, y.w & km1b), bf.x, bf.y);
        }
      }
    }
    // ---- scores, value exponents, reference maximum
    const float4 a4k = *reinterpret_cast<const float4*>(ak + tq);
    const float4 a4v = *reinterpret_cast<const float4*>(av + tq);
    const float akv[4] = {a4k.x, a4k.y, a4k.z, a4k.w};
    const float avv[4] = {a4v.x, a4v.y, a4v.z, a4v.w};
    const int tg = (tile_lo + ti) * TILE + tq;
    bool ok[4];
    float lg[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      ok[k] = tg + k >= t_lo && tg + k < t_end;
      // floor(log2 alpha^V) from the exponent field (>= -64; 0 and subnormals -> -64)
      lg[k] = static_cast<float>(max(static_cast<int>((__float_as_uint(avv[k]) >> 23) & 0xFF) - 127, -64));
    }
    float sc4[NP][4];
    bool over = false;
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      const float r[4] = {kacc[0][p][0] + kacc[0][p][1], kacc[0][p][2] + kacc[0][p][3],
                          kacc[1][p][0] + kacc[1][p][1], kacc[1][p][2] + kacc[1][p][3]};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        sc4[p][k] = ok[k] ? akv[k] * fmaf(r[k], sg[p], -cg[p]) : -INFINITY;
        over |= sc4[p][k] + lg[k] > mrun[p] + 8.0f;
      }
    }
    if (__any_sync(0xffffffffu, over)) {
      // a token exceeds the reference by more than 2^8: raise it to the tile's maximum
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        float e = fmaxf(fmaxf(sc4[p][0] + lg[0], sc4[p][1] + lg[1]), fmaxf(sc4[p][2] + lg[2], sc4[p][3] + lg[3]));
        e = fmaxf(e, __shfl_xor_sync(0xffffffffu, e, 4));
        e = fmaxf(e, __shfl_xor_sync(0xffffffffu, e, 8));
        e = fmaxf(e, __shfl_xor_sync(0xffffffffu, e, 16));
        if (e > mrun[p]) {
          const float f = fast_exp2(mrun[p] - e);                  // mrun = -inf -> 0
          lsum[p] *= f;
          ssum[p] *= f;
#pragma unroll
          for (int jj = 0; jj < NJ; ++jj)
#pragma unroll
            for (int z = 0; z < 4; ++z) vacc[jj][p][z] *= f;
          mrun[p] = e;
        }
      }
    }
    // ---- P' = 2^(s - m) alpha^V (times 2^5 into f16 range) as f16 hi / lo value B fragments:
    // token quad g of the warp is value k-step g >> 2, fragment lane column t' = g & 3, with
    // registers b0 = (token 0, token 2), b1 = (token 1, token 3) in columns 2t (hi) and 2t + 1 (lo)
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      float pv[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float pk = ok[k] ? fast_exp2(sc4[p][k] - mrun[p]) : 0.0f;
        // masked tokens may hold any bits in alpha (beyond the context): select, never multiply
        pv[k] = ok[k] ? pk * avv[k] * kPScale : 0.0f;
        lsum[p] += pk;
      }
      ssum[p] += (pv[0] + pv[1]) + (pv[2] + pv[3]);
      const __half2 h02 = __floats2half2_rn(pv[0], pv[2]), h13 = __floats2half2_rn(pv[1], pv[3]);
      const float2 f02 = __half22float2(h02), f13 = __half22float2(h13);
      const __half2 l02 = __floats2half2_rn(pv[0] - f02.x, pv[2] - f02.y);
      const __half2 l13 = __floats2half2_rn(pv[1] - f13.x, pv[3] - f13.y);
      uint2* dst = reinterpret_cast<uint2*>(pfw) + ((g >> 2) * NP + p) * 32 + (g & 3);
      dst[4 * (2 * t)] = make_uint2(*reinterpret_cast<const uint32_t*>(&h02), *reinterpret_cast<const uint32_t*>(&h13));
      dst[4 * (2 * t + 1)] = make_uint2(*reinterpret_cast<const uint32_t*>(&l02), *reinterpret_cast<const uint32_t*>(&l13));
    }
    __syncwarp();
    // ---- values: M-tile rows are record entries, K = the 16 tokens of k-step kv (quads
    // 8 wq + 4 kv + t); lane t's K columns 2t, 2t + 1 are tokens 0, 2 of its quad (bytes 0, 2 of
    // a slot word), 2t + 8, 2t + 9 tokens 1, 3 (bytes 1, 3, shifted down)
#pragma unroll
    for (int kv = 0; kv < 2; ++kv) {
      uint2 bf[NP];
#pragma unroll
      for (int p = 0; p < NP; ++p) bf[p] = reinterpret_cast<const uint2*>(pfw)[(kv * NP + p) * 32 + lane];
      const uint32_t* vq = vt + 4 * (8 * wq + 4 * kv + t);
#pragma unroll
      for (int jw = 0; jw < N2W; ++jw) {
        const uint2 xx = *reinterpret_cast<const uint2*>(vq + jw * TILE + d2off);
        const uint4 af = make_uint4(xx.x & vm2, xx.y & vm2, (xx.x >> 8) & vm2, (xx.y >> 8) & vm2);
#pragma unroll
        for (int p = 0; p < NP; ++p) mma_f16(vacc[jw][p], af, bf[p].x, bf[p].y);
      }
#pragma unroll
      for (int u = 0; u < N1W; ++u) {
        const uint4 s4 = *reinterpret_cast<const uint4*>(vq + (N2W + u) * TILE);
        const uint4 afa = make_uint4(s4.x & vm1, s4.z & vm1, (s4.x >> 8) & vm1, (s4.z >> 8) & vm1);  // fields 0..15
        const uint4 afb = make_uint4(s4.y & vm1, s4.w & vm1, (s4.y >> 8) & vm1, (s4.w >> 8) & vm1);  // 16..31
#pragma unroll
        for (int p = 0; p < NP; ++p) {
          mma_f16(vacc[N2W + 2 * u][p], afa, bf[p].x, bf[p].y);
          mma_f16(vacc[N2W + 2 * u + 1][p], afb, bf[p].x, bf[p].y);
        }
      }
    }
    __syncwarp();
    // ---- release the stage; the last of the group's four warps refills it
    if (lane == 0) {
      __threadfence_block();
      const int old = atomicAdd(cnt + s, 1);
      if ((old & 3) == 3 && j + NS < n_j) {
        __threadfence_block();
        ptx::fence_proxy_async_smem();
        issue(j + NS, s);
      }
    }
    if (++s == NS) {
      s = 0;
      ph ^= 1;
    }
  }

  __syncthreads();
  if (s_abort) {
    // a wait gave up: let every copy still in flight land (bounded) before leaving
    if (leader)
      for (int j = max(0, s_issued[wg] - NS); j < s_issued[wg]; ++j)
        ptx::mbar_wait_sleep(full + j % NS, (j / NS) & 1, &s_never, 20);
    return;
  }
  // ---- per-warp (m, l, S') and entry sums into the drained rings
  float* epi = reinterpret_cast<float*>(smb + L.ring);
  const int NE = a.n_entries, NEP = fused_entry_pitch(NE);
  constexpr int kEpiStride = 3 * MAX_GROUP;                  // + GMAX * NEP floats per warp
  const int wstride = kEpiStride + GMAX * NEP;               // per-warp block: (m, l, S'), then E
  float* wm = epi + warp * wstride;                          // [m, l, S'][MAX_GROUP], then E[GMAX][NEP]
  float* wE = wm + kEpiStride;
#pragma unroll
  for (int p = 0; p < NP; ++p) {
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      lsum[p] += __shfl_xor_sync(0xffffffffu, lsum[p], o);
      ssum[p] += __shfl_xor_sync(0xffffffffu, ssum[p], o);
    }
    if (lane < 4) {
      const int q = 4 * p + lane;
      wm[q] = mrun[p];
      wm[MAX_GROUP + q] = lsum[p];
      wm[2 * MAX_GROUP + q] = ssum[p] * (1.0f / kPScale);
    }
  }
  {
    // lane (g, t) holds entry rows g (c0 + c1) and g + 8 (c2 + c3) of every M-tile for query
    // 4p + t; raw sums times 2^24 / (row scale) / 2^5 = sum P' digit
#pragma unroll
    for (int jj = 0; jj < NJ; ++jj) {
      int e;
      float sc;
      if (jj < N2W) {
        e = 16 * jj + g;
        sc = pow2i(19 - 2 * (g & 3));
      } else {
        const int u = (jj - N2W) >> 1, half = (jj - N2W) & 1;
        e = 16 * N2W + 32 * u + 16 * half + g;
        sc = pow2i(19 - g);
      }
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        float* dst = wE + (4 * p + t) * NEP;
        if (e < NE) dst[e] = (vacc[jj][p][0] + vacc[jj][p][1]) * sc;
        if (e + 8 < NE) dst[e + 8] = (vacc[jj][p][2] + vacc[jj][p][3]) * sc;
      }
    }
  }
  __syncthreads();
  // ---- the CTA maximum M per query, each warp's factor 2^(m_w - M) and the totals l and S'
  // (warp q, lane w = warp w's values), then the entry sums over the warps (each warp's sums
  // scaled once, in a fixed order)
  float* ff = epi + NW * wstride;                            // [NW][GMAX]
  float* tot = ff + NW * GMAX;                               // [M, l, S'][GMAX]
  float* etot = tot + 3 * GMAX;                              // [GMAX][NEP]
  if (warp < GMAX) {
    const float* ww = epi + (lane < NW ? lane : 0) * wstride;
    const float mw = lane < NW ? ww[warp] : -INFINITY;
    float M = mw;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float f = mw > -INFINITY ? fast_exp2(mw - M) : 0.0f;
    float l = lane < NW ? f * ww[MAX_GROUP + warp] : 0.0f;
    float sp = lane < NW ? f * ww[2 * MAX_GROUP + warp] : 0.0f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      l += __shfl_xor_sync(0xffffffffu, l, o);
      sp += __shfl_xor_sync(0xffffffffu, sp, o);
    }
    if (lane < NW) ff[lane * GMAX + warp] = f;
    if (lane == 0) {
      tot[warp] = M;
      tot[GMAX + warp] = l;
      tot[2 * GMAX + warp] = sp;
    }
  }
  __syncthreads();
  for (int i4 = tid; i4 < GMAX * NEP / 4; i4 += NT) {         // four entries of one query row
    const int idx = 4 * i4, q = idx / NEP;
    float4 ev[NW];
    float fw[NW];
#pragma unroll
    for (int w = 0; w < NW; ++w) {                           // all loads first, then the sums
      ev[w] = *reinterpret_cast<const float4*>(epi + w * wstride + kEpiStride + idx);
      fw[w] = ff[w * GMAX + q];
    }
    float4 e0 = make_float4(0.0f, 0.0f, 0.0f, 0.0f), e1 = e0;
#pragma unroll
    for (int w = 0; w < NW; w += 2) {
      e0.x = fmaf(fw[w], ev[w].x, e0.x); e0.y = fmaf(fw[w], ev[w].y, e0.y);
      e0.z = fmaf(fw[w], ev[w].z, e0.z); e0.w = fmaf(fw[w], ev[w].w, e0.w);
      e1.x = fmaf(fw[w + 1], ev[w + 1].x, e1.x); e1.y = fmaf(fw[w + 1], ev[w + 1].y, e1.y);
      e1.z = fmaf(fw[w + 1], ev[w + 1].z, e1.z); e1.w = fmaf(fw[w + 1], ev[w + 1].w, e1.w);
    }
    *reinterpret_cast<float4*>(etot + idx) = make_float4(e0.x + e1.x, e0.y + e1.y, e0.z + e1.z, e0.w + e1.w);
  }
  __syncthreads();
  // ---- the split's partial per query: thread = (value channel c, query parity part)
  const size_t pbase = (static_cast<size_t>(b) * a.n_q + head * G) * a.n_splits;
  {
    const uint4 cev = *reinterpret_cast<const uint4*>(cetab + c * 8);
    const uint32_t cw4[4] = {cev.x, cev.y, cev.z, cev.w};
    const float4 wa = *reinterpret_cast<const float4*>(cw8 + c * 8), wb = *reinterpret_cast<const float4*>(cw8 + c * 8 + 4);
    const float w8[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
    int e8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) e8[k] = static_cast<int>(cw4[k >> 1] >> (16 * (k & 1))) & 0xFFFF;   // entry k of c
    const float off = reinterpret_cast<const float*>(smb + L.qc)[2 * MAX_GROUP + c];
    for (int q = part; q < G; q += WG) {
      float o = -off * tot[2 * GMAX + q];
#pragma unroll
      for (int k = 0; k < 8; ++k) o = fmaf(w8[k], etot[q * NEP + e8[k]], o);
      float* dst = a.ws + (pbase + static_cast<size_t>(q) * a.n_splits + split) * a.pstride;
      dst[c] = o;
      if (c == 0) {
        dst[D] = tot[q];
        dst[D + 1] = tot[GMAX + q];
      }
    }
  }
}

// Merge of the splits of one (sequence, query head): M = max_s m_s, w_s = 2^(m_s - M),
// o_c = sum_s w_s o_{s,c}, l = sum_s w_s l_s, o_hat_c = o_c f^V_c, out = U_V o_hat / l.
// Uncompressed tokens (the full-precision sink and recent window of Sec. 6) join the same
// softmax here: their scores q.k/sqrt(128), weights 2^(s - m_f) and sum_t p_t v_t are taken in
// the original basis and merged with the packed part by log-sum-exp.
// Launched as a programmatic dependent of the split kernel: U_V^T (a plan constant) is staged
// while the splits finish; the partials are read only after the grid dependency resolves.
constexpr int kMThreads = 512;
constexpr int kMWarps = kMThreads / 32;

__global__ void __launch_bounds__(kMThreads)
    aatc_decode_merge_kernel(const DecodeArgs a) {
  extern __shared__ __align__(16) float ms[];
  float* ut_s = ms;                                  // [128 c][128 d]
  float* osum = ut_s + D * D;                        // [kMWarps][128]
  float* ohat = osum + kMWarps * D;                  // [128]
  float* sf = ohat + D;                              // [n_full] scores, then weights, of full tokens
  __shared__ float red[2][kMWarps];
  __shared__ uint64_t bar;
  __shared__ int s_abort;
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int head = j / a.group;
  const int sv = (a.layer * a.n_kv + head) * 2 + 1;
  if (tid == 0) {
    s_abort = 0;
    ptx::mbar_init(&bar, 1);
    ptx::fence_mbar_init();
    ptx::mbar_arrive_expect_tx(&bar, D * D * 4);
    ptx::bulk_load(ut_s, a.u32t + static_cast<size_t>(sv) * D * D, D * D * 4, &bar);
  }
  // the next call's query kernel may start its plan-constant prologue now; it reads the query
  // and the workspace only after this grid has completed (its griddepcontrol.wait)
  ptx::grid_launch_dependents();
  const float fv = tid < D ? a.f[sv * D + tid] : 0.0f;
  // ---- uncompressed tokens (inputs of this call, not produced by the split kernel)
  float m_f = -INFINITY, l_f = 0.0f;
  float of = 0.0f;                                   // thread d < 128: sum_t p_t v_t[d]
  if (a.n_full > 0) {
    // q and the full tokens were complete before the query kernel let the split kernel start;
    // with no packed range this kernel follows the caller's grid directly
    if (a.n_splits == 0) ptx::grid_dependency_wait();
    const float scale = kLog2e * 0.08838834764831845f;
    const uint2 qq = *reinterpret_cast<const uint2*>(a.q + (static_cast<size_t>(b) * a.n_q + j) * D + 4 * lane);
    const float2 q01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qq.x));
    const float2 q23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qq.y));
    float mloc = -INFINITY;
    for (int t = warp; t < a.n_full; t += kMWarps) {
      const size_t row = ((static_cast<size_t>(b) * a.full_cap + t) * a.n_kv + head) * D;
      const uint2 kk = *reinterpret_cast<const uint2*>(a.k_full + row + 4 * lane);
      const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kk.x));
      const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kk.y));
      float d = fmaf(q01.x, k01.x, fmaf(q01.y, k01.y, fmaf(q23.x, k23.x, q23.y * k23.y)));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
      if (lane == 0) sf[t] = d * scale;
      mloc = fmaxf(mloc, d * scale);
    }
    if (lane == 0) red[0][warp] = mloc;
    __syncthreads();
    m_f = red[0][0];
#pragma unroll
    for (int w = 1; w < kMWarps; ++w) m_f = fmaxf(m_f, red[0][w]);
    float lp = 0.0f;
    for (int t = tid; t < a.n_full; t += kMThreads) {
      const float pw = fast_exp2(sf[t] - m_f);
      sf[t] = pw;
      lp += pw;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lp += __shfl_xor_sync(0xffffffffu, lp, o);
    if (lane == 0) red[1][warp] = lp;
    __syncthreads();
    l_f = 0.0f;
#pragma unroll
    for (int w = 0; w < kMWarps; ++w) l_f += red[1][w];
    {
      // four threads per dimension, tokens t = quarter (mod 4)
      const int d = tid & (D - 1), qtr = tid >> 7;
      float acc = 0.0f;
      for (int t = qtr; t < a.n_full; t += 4)
        acc = fmaf(sf[t], __bfloat162float(a.v_full[((static_cast<size_t>(b) * a.full_cap + t) * a.n_kv + head) * D + d]), acc);
      osum[qtr * D + d] = acc;
    }
    __syncthreads();
    if (tid < D) of = (osum[tid] + osum[D + tid]) + (osum[2 * D + tid] + osum[3 * D + tid]);
    __syncthreads();
  }
  // ---- packed splits: warp w merges splits w, w + 16, ... online (running max, rescaled sums),
  // eight splits' loads in flight per round; then the 16 warp partials are merged per channel.
  float M = -INFINITY, L = 0.0f;
  if (a.n_splits > 0) {
    ptx::grid_dependency_wait();                     // the split kernel's partials
    const float* src = a.ws + (static_cast<size_t>(b) * a.n_q + j) * a.n_splits * a.pstride;
    float mw = -INFINITY, lw = 0.0f;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    for (int s0 = warp; s0 < a.n_splits; s0 += kMWarps * 8) {
      float2 ml[8];
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int s = s0 + kMWarps * u;
        if (s < a.n_splits) {
          ml[u] = __ldcg(reinterpret_cast<const float2*>(src + static_cast<size_t>(s) * a.pstride + D));
          v[u] = __ldcg(reinterpret_cast<const float4*>(src + static_cast<size_t>(s) * a.pstride + 4 * lane));
        } else {
          ml[u] = make_float2(-INFINITY, 0.0f);
          v[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        }
      }
      float mc = mw;
#pragma unroll
      for (int u = 0; u < 8; ++u) mc = fmaxf(mc, ml[u].x);
      if (mc > -INFINITY) {                          // else nothing attended so far: sums stay 0
        const float r = fast_exp2(mw - mc);              // mw = -inf -> 0
        lw *= r;
        acc.x *= r; acc.y *= r; acc.z *= r; acc.w *= r;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float w = fast_exp2(ml[u].x - mc);
          lw = fmaf(w, ml[u].y, lw);
          acc.x = fmaf(w, v[u].x, acc.x);
          acc.y = fmaf(w, v[u].y, acc.y);
          acc.z = fmaf(w, v[u].z, acc.z);
          acc.w = fmaf(w, v[u].w, acc.w);
        }
        mw = mc;
      }
    }
    *reinterpret_cast<float4*>(osum + warp * D + 4 * lane) = acc;
    if (lane == 0) {
      red[0][warp] = mw;
      red[1][warp] = lw;
    }
    __syncthreads();
#pragma unroll
    for (int w = 0; w < kMWarps; ++w) M = fmaxf(M, red[0][w]);
    if (M > -INFINITY)
#pragma unroll
      for (int w = 0; w < kMWarps; ++w) L = fmaf(fast_exp2(red[0][w] - M), red[1][w], L);
  }
  // ---- log-sum-exp merge of the two parts: out = (U_V (f o) a_p + o_f a_f) / (L a_p + l_f a_f)
  const float Mt = fmaxf(M, m_f);
  const float ap = a.n_splits > 0 ? fast_exp2(M - Mt) : 0.0f;
  const float af = a.n_full > 0 ? fast_exp2(m_f - Mt) : 0.0f;
  const float inv_den = 1.0f / fmaf(L, ap, l_f * af);
  if (tid < D) {
    float o = 0.0f;
    if (a.n_splits > 0 && M > -INFINITY) {
#pragma unroll
      for (int w = 0; w < kMWarps; ++w) o = fmaf(fast_exp2(red[0][w] - M), osum[w * D + tid], o);
    }
    ohat[tid] = o * fv * ap;
  }
  if (!ptx::mbar_wait_sleep(&bar, 0, &s_abort, 100)) atomicOr(a.err, 2);
  __syncthreads();
  // out[d] = sum_c U_V[d][c] o_hat[c]: four threads per dimension, quarters of c
  {
    const int d = tid & (D - 1), qtr = tid >> 7;
    float r4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int c = 0; c < 32; ++c) r4[c & 3] = fmaf(ut_s[(qtr * 32 + c) * D + d], ohat[qtr * 32 + c], r4[c & 3]);
    osum[qtr * D + d] = (r4[0] + r4[1]) + (r4[2] + r4[3]);
  }
  __syncthreads();
  if (tid < D)
    a.out[(static_cast<size_t>(b) * a.n_q + j) * D + tid] =
        ((osum[tid] + osum[D + tid]) + (osum[2 * D + tid] + osum[3 * D + tid]) + of * af) * inv_den;
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

// bf16 tiles of 128 tokens x 128 dims in a ring of three, 256 B rows with the 16-byte chunks
// XOR-swizzled by the row (chunk c of row r at chunk c ^ (r & 7)): the row-per-thread 128-bit
// reads of the score pass and the row-shared 64-bit reads of the value pass are both free of
// bank conflicts without padding.
constexpr int kB16Stages = 3;
constexpr int kB16Tile = TILE * D;                         // bf16 elements per tile

template <int GP>
__global__ void __launch_bounds__(kThreads)
    aatc_bf16_split_kernel(const Bf16Args a) {
  extern __shared__ __align__(16) float sm[];
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int G = a.group;
  float* qs = sm;                                          // [128][GP]
  float* red = qs + D * GP;                                // [32]
  float* sc = red + 32;                                    // [split_len][GP]
  __nv_bfloat16* ring = reinterpret_cast<__nv_bfloat16*>(sc + a.split_len * GP);   // [3][128][128]
  float* accs = reinterpret_cast<float*>(ring);            // [4][GP][128], over the drained ring
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE;
  const int tile_lo = static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const int t_begin = tile_lo * TILE;
  const int t_end = min(a.n_ctx, tile_hi * TILE);
  const int n_tiles_split = tile_hi - tile_lo;
  const int n_seq = 2 * n_tiles_split;                     // key tiles, then value tiles
  const float scale = kLog2e * 0.08838834764831845f;
  for (int i = tid; i < GP * D; i += kThreads) {
    const int g = i / D, d = i % D;
    qs[d * GP + g] =
        g < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + g) * D + d]) * scale : 0.0f;
  }
  const int tile0 = t_begin / TILE;
  auto stage_seq = [&](int i) {                            // tile i of the sequence into buffer i % 3
    const __nv_bfloat16* base = i < n_tiles_split ? a.k : a.v;
    const int tile = tile0 + (i < n_tiles_split ? i : i - n_tiles_split);
    __nv_bfloat16* dst = ring + (i % kB16Stages) * kB16Tile;
    for (int e = tid; e < TILE * 16; e += kThreads) {
      const int r = e >> 4, ch = e & 15;
      const int t = min(tile * TILE + r, a.n_ctx - 1);     // padding rows: a valid token, masked later
      cp_async16(dst + r * D + ((ch ^ (r & 7)) << 3),
                 base + ((static_cast<size_t>(b) * a.max_tokens + t) * a.n_kv + head) * D + ch * 8);
    }
    cp_async_commit();
  };
  // before tile i: it has landed (tile i + 1 may still be in flight), every thread is past tile
  // i - 1, and tile i + 2 goes into the buffer tile i - 1 used
  auto next_tile = [&](int i) {
    if (i + 1 < n_seq) cp_async_wait_one(); else cp_async_wait_all();
    __syncthreads();
    if (i + 2 < n_seq) stage_seq(i + 2);
    return ring + (i % kB16Stages) * kB16Tile;
  };
  stage_seq(0);
  if (n_seq > 1) stage_seq(1);
  __syncthreads();                                         // query columns visible
  float mloc[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) mloc[g] = -INFINITY;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const __nv_bfloat16* row = next_tile(ti) + tid * D;   // thread = token tid of the tile
    float s[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) s[g] = 0.0f;
#pragma unroll 4
    for (int c = 0; c < 16; ++c) {
      float kv[8];
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(row + ((c ^ (tid & 7)) << 3)), kv);
      const int d0 = 8 * c;
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
  __syncthreads();
  block_reduce<GP, true>(mloc, red);
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
  const int dch = dg >> 1, dsub = 4 * (dg & 1);            // dims 4 dg .. 4 dg + 3: chunk, position
  float acc[GP][4];
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[g][i] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const __nv_bfloat16* vt = next_tile(n_tiles_split + ti);
    const int tend = min(TILE, t_end - (tile0 + ti) * TILE);
    for (int tt = tq; tt < tend; tt += 4) {
      const uint2 r = *reinterpret_cast<const uint2*>(vt + tt * D + ((dch ^ (tt & 7)) << 3) + dsub);
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
  __syncthreads();                                         // ring drained: accs may overwrite it
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
  auto rec_word = [&](int w) -> uint32_t {
    const uint32_t* ww = tile + static_cast<size_t>(w) * TILE;
    if (kind == 0) return ww[tt];
    const int q4 = 4 * (tt >> 2), sh = 8 * (tt & 3);
    const uint32_t b0 = (ww[q4 + 0] >> sh) & 0xFFu, b1 = (ww[q4 + 2] >> sh) & 0xFFu;
    const uint32_t b2 = (ww[q4 + 1] >> sh) & 0xFFu, b3 = (ww[q4 + 3] >> sh) & 0xFFu;
    return b0 | (b1 << 8) | (b2 << 16) | (b3 << 24);
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

// Launch with programmatic stream serialization: the kernel may start before the preceding
// grid in the stream completes; it synchronizes with griddepcontrol.wait before touching
// anything that grid produces.
template <typename... Args>
cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <int JPW, int NP>
cudaError_t launch_split_t(const DecodeArgs& a, int batch, size_t smem, cudaStream_t st) {
  cudaError_t e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_decode_split_kernel<JPW, NP>), smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(aatc_decode_split_kernel<JPW, NP>, dim3(a.n_splits, a.n_kv, batch), dim3(kThreads), smem, st, a);
}

template <int NP>
cudaError_t launch_split_g(const DecodeArgs& a, int batch, int jpw, size_t smem, cudaStream_t st) {
  if (jpw <= 4) return launch_split_t<4, NP>(a, batch, smem, st);
  if (jpw <= 8) return launch_split_t<8, NP>(a, batch, smem, st);
  return launch_split_t<12, NP>(a, batch, smem, st);
}

template <int GP>
cudaError_t launch_bf16_split(const Bf16Args& a, int batch, cudaStream_t st) {
  const size_t smem = bf16_split_smem(GP, a.split_len);
  cudaError_t e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_bf16_split_kernel<GP>), smem);
  if (e != cudaSuccess) return e;
  aatc_bf16_split_kernel<GP><<<dim3(a.n_splits, a.n_kv, batch), kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

// Record shape shared by every key and value stream of `layer` (D2 words, D1 words), or false.
static bool layer_shape(const Plan& plan, int layer, int* n2w, int* n1w) {
  const int hk = plan.dims.n_kv_heads;
  for (int s = 0; s < 2 * hk; ++s) {
    const StreamLayout& l = plan.layout[layer * 2 * hk + s];
    const int a = l.n2 / 16, b = (l.n1 + 31) / 32;
    if (s == 0) {
      *n2w = a;
      *n1w = b;
    } else if (a != *n2w || b != *n1w) {
      return false;
    }
  }
  return true;
}

using FusedKernel = void (*)(const DecodeArgs);

// The record shapes the fused kernel is built for: (D2 words, D1 words) of the per-stream plans at
// 1.5, 2, 2.75 and 4 bits per channel.
// Warp groups per CTA (one CTA per SM): four for up to four query heads per kv-head (16 warps, at
// most 128 registers), two for five to eight (twice the value accumulators).
template <int NP>
constexpr int fused_groups() { return NP == 1 ? 4 : 2; }

template <int NP>
static FusedKernel fused_kernel_for(int n2w, int n1w) {
  constexpr int WG = fused_groups<NP>();
  if (n2w == 9 && n1w == 2) return aatc_decode_fused_kernel<9, 2, NP, WG>;
  if (n2w == 3 && n1w == 3) return aatc_decode_fused_kernel<3, 3, NP, WG>;
  if (n2w == 5 && n1w == 3) return aatc_decode_fused_kernel<5, 3, NP, WG>;
  if (n2w == 13 && n1w == 3) return aatc_decode_fused_kernel<13, 3, NP, WG>;
  return nullptr;
}

cudaError_t launch_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                          int max_tokens, float* out, void* ws, cudaStream_t st, const DecodeExtra& extra) {
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
  a.t_first = extra.t_first;
  a.k_full = static_cast<const __nv_bfloat16*>(extra.k_full);
  a.v_full = static_cast<const __nv_bfloat16*>(extra.v_full);
  a.n_full = extra.n_full;
  a.full_cap = extra.full_cap;
  const int np = (a.group + 3) / 4;
  // the fused kernel: a packed range and one record shape (uncompressed tokens, if any, join in
  // the merge kernel)
  int n2w = 0, n1w = 0;
  FusedKernel fk = nullptr;
  if (extra.t_first < n_ctx && plan.max_bits <= 8 && layer_shape(plan, layer, &n2w, &n1w))
    fk = np == 1 ? fused_kernel_for<1>(n2w, n1w) : fused_kernel_for<2>(n2w, n1w);
  const int range = n_ctx - (extra.t_first / TILE) * TILE;
  const DecodeSplit sp = decode_split_for(batch, a.n_kv, range, plan.num_sms, fk != nullptr);
  a.n_splits = extra.t_first < n_ctx ? sp.n_splits : 0;     // no packed range: merge kernel only
  a.split_len = sp.split_len;
  {
    const long n_cta = static_cast<long>(sp.n_splits) * a.n_kv * batch;
    a.num_sms = plan.num_sms;
    a.cta_per_sm = plan.num_sms > 0 && n_cta % plan.num_sms == 0 ? static_cast<int>(n_cta / plan.num_sms) : 0;
  }
  const DecodeWs wsl = decode_ws_layout(batch, a.n_q, a.n_kv, plan.n_entries, plan.n_words, sp);
  a.pstride = wsl.pstride;
  a.ks_stride = wsl.ks_stride;
  a.qfrag = reinterpret_cast<uint4*>(static_cast<char*>(ws) + wsl.qfrag_off);
  a.qcorr = reinterpret_cast<float*>(static_cast<char*>(ws) + wsl.qcorr_off);
  if (plan.n_entries > kMaxEntries) return cudaErrorNotSupported;
  // every shape refusal comes before the first launch of the call
  const size_t msm = 4 * (static_cast<size_t>(D) * D + kMWarps * D + D + static_cast<size_t>((a.n_full + 3) & ~3));
  if (msm > 227 * 1024) return cudaErrorNotSupported;
  cudaError_t e = cudaSuccess;
  if (fk) {
    const int wu = n2w + n1w, nks = n2w + 2 * n1w;
    const int wg = np == 1 ? fused_groups<1>() : fused_groups<2>();
    // the deepest ring (up to 3 stages per warp group) that fits the shared memory of one SM
    size_t smem = 0;
    for (a.n_stages = 3; a.n_stages >= 2; --a.n_stages) {
      smem = static_cast<size_t>(FusedSmem(wu, nks, np, wg, plan.n_entries, a.n_stages).total);
      if (smem <= 227 * 1024) break;
    }
    if (a.n_stages < 2) return cudaErrorNotSupported;
    e = ensure_smem_optin(reinterpret_cast<const void*>(fk), smem);
    if (e != cudaSuccess) return e;
    const unsigned n_cta = static_cast<unsigned>(static_cast<long>(sp.n_splits) * a.n_kv * batch);
    e = launch_pdl(fk, dim3(n_cta), dim3(128 * wg), smem, st, a);
    if (e != cudaSuccess) return e;
    e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_decode_merge_kernel), msm);
    if (e != cudaSuccess) return e;
    return launch_pdl(aatc_decode_merge_kernel, dim3(a.n_q, batch), dim3(kMThreads), msm, st, a);
  }
  // largest key k-step count and value word count over the layer's streams
  int n_ks = 1, n_jobs_v = 1;
  for (int h = 0; h < a.n_kv; ++h) {
    const StreamLayout& lk = plan.layout[(layer * a.n_kv + h) * 2];
    const StreamLayout& lv = plan.layout[(layer * a.n_kv + h) * 2 + 1];
    n_ks = std::max(n_ks, lk.n2 / 16 + 2 * ((lk.n1 + 31) / 32));
    n_jobs_v = std::max(n_jobs_v, lv.n2 / 16 + 2 * ((lv.n1 + 31) / 32));
  }
  const SplitSmem L(n_ks, np, sp.split_len, plan.n_words, plan.n_entries);
  const size_t smem = static_cast<size_t>(L.total);
  const int jpw = (n_jobs_v + kWarps - 1) / kWarps;            // value M-tiles per warp
  if (a.n_splits > 0 && (jpw > 12 || smem > 227 * 1024)) return cudaErrorNotSupported;
  if (a.n_splits > 0) {
    e = launch_pdl(aatc_decode_query_kernel, dim3(a.n_kv, batch, MAX_GROUP), dim3(kQThreads), 0, st, a);
    if (e != cudaSuccess) return e;
    e = np == 1 ? launch_split_g<1>(a, batch, jpw, smem, st) : launch_split_g<2>(a, batch, jpw, smem, st);
    if (e != cudaSuccess) return e;
  }
  e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_decode_merge_kernel), msm);
  if (e != cudaSuccess) return e;
  return launch_pdl(aatc_decode_merge_kernel, dim3(a.n_q, batch), dim3(kMThreads), msm, st, a);
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

size_t bf16_split_smem(int gp, int split_len) {
  // query columns [128][gp], reduction scratch, scores [split_len][gp] (fp32); a ring of three
  // bf16 tiles [128][128], which the per-quarter sums [4][gp][128] reuse at the end
  return 4 * (static_cast<size_t>(D) * gp + 32 + static_cast<size_t>(split_len) * gp) +
         static_cast<size_t>(kB16Stages) * TILE * D * 2;
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
  if (plan->dims.n_q_heads / plan->dims.n_kv_heads > MAX_GROUP || plan->group_heads > 1) return AATC_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(cache) & 15u) != 0) return AATC_ERR_INVALID_ARG;
  if (decode_workspace_for(*plan, batch, n_ctx) > AATC_NOALLOC_SCRATCH_BYTES) return AATC_ERR_WORKSPACE;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return status_from_cuda(e);
  if (dev != plan->device) return AATC_ERR_INVALID_ARG;       // the array used is the current device's
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
  return status_from_cuda(launch_decode(*plan, layer, q, cache, batch, n_ctx, max_tokens, out, scratch,
                                        static_cast<cudaStream_t>(stream), DecodeExtra{}));
}
