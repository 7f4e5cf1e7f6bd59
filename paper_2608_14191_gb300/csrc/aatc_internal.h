// Internal declarations shared by the C ABI (capi.cpp), the planner and the CUDA kernels.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>

#include <cuda_runtime.h>

#include "aatc.h"

#if defined(__CUDACC__)
#define AATC_HD __host__ __device__
#else
#define AATC_HD
#endif

namespace aatc {

constexpr int D = 128;              // head_dim
constexpr int TILE = 128;           // tokens per word-planar cache tile
constexpr int MAX_GROUP = 8;        // query heads per kv-head supported by the decode kernels
constexpr uint32_t PLAN_MAGIC = 0xAA7C0DE1u;
constexpr uint32_t PLAN_DEAD = 0xDEADDEADu;

// Per-channel encode constants (one 16-byte load in the encode epilogue).
struct ChanEnc {
  float inv_f;            // 1 / f_c, f_c = s_c 2^(1-b_c); 0 for dropped channels
  float hi;               // 2^(b_c-1) - 1 as float: upper clamp of h/Delta + 1/2 (0 for dropped)
  float magic;            // 1.5 * 2^23 + 2^(b_c-1): round-down add leaves u = code + 2^(b-1) in the mantissa
  float off;              // 2^(b_c-1) (offset of the stored code), 0 for dropped
};

// Record layout of one stream.  The stored value u = code + 2^(b-1) of every retained channel
// is split into base-4 digits and single top bits:
//   D2: for k = 0..7, digit k (bits 2k, 2k+1) of channels 0..l2[k]-1  (16 two-bit fields/word)
//   D1: the top bit of every odd-width channel (channel order), then the digits that did not
//       fill the last D2 word, each as two single bits (32 one-bit fields/word)
// Record words: n2/16 D2 words, then ceil(n1/32) D1 words, then zeros up to the plan's W.
// `entry[e]` (int16, per stream) lists the D2 entries then the D1 entries as
// (channel | bit shift << 8); padding entries are -1.
struct StreamLayout {
  int n2;                 // D2 entries (a multiple of 16)
  int n1;                 // D1 entries
  int words;              // record words this stream uses
  int nret;               // retained channels R
  int l2[8];              // D2 digit-layer lengths (digits kept in D2)
  int l2all[8];           // channels with b >= 2k + 2 (digit k exists; those past l2[k] moved to D1)
  int lodd[8];            // channels with b >= 2k + 1 (width 2k + 1 channels: [l2all[k], lodd[k]))
};

// Record entries of one channel: at most 8 digits, or 7 with one moved to D1 as two bits plus an
// odd top bit, so 9 at 16 bits; the per-channel entry table keeps kChanEnt slots.
constexpr int kChanEnt = 16;
// The register-resident encode keeps the high bytes of the first 32 stored values: channels
// wider than 8 bits must lie in that prefix (widths are non-increasing in storage order).
constexpr int kMaxWideChannels = 32;

struct PlanDevice {
  const void* ubf16_t;    // bf16 [S][128 channel][128 dim]   encode basis (MMA B operand, K-major)
  const float* u32;       // fp32 [S][128 dim][128 channel]   decode query rotation
  const float* u32t;      // fp32 [S][128 channel][128 dim]   decode inverse value transform
  const ChanEnc* enc;     // [S][128]
  const float* inv_s;     // [S][128] 1/s_c (0 for dropped)
  const float* f;         // [S][128] f_c (0 for dropped)
  const StreamLayout* lay;  // [S]
  const short* entry;     // [S][n_entries]
  const short* chan_ent;  // [S][128][8]: entries of each channel (-1 padded)
  int* err;               // [4] sticky device flags
};

// Head-group plans (one transform over the n = 128 g_h channels of g_h kv-heads, Sec. 5 Step 1):
// a group stream is kept as g_h slice streams in the per-kv-head slots (layer, g g_h + s, K|V) of
// the plan tables and of the cache; slice s holds the group's storage-order channels s, s + g_h,
// s + 2 g_h, ... (widths stay non-increasing in every slice) and all slices of a token share one
// alpha, written to every slice's slot.  Group tables, channels in slice-major order
// (j' = 128 s + c for storage channel j = c g_h + s):
struct GroupDevice {
  const void* ubf;        // bf16 [L][n_groups][2][n channel][n dim]   encode operand (K-major)
  const float* uk;        // fp32 [L][n_groups][n dim][n channel]      key rotation U_K
  const float* uvt;       // fp32 [L][n_groups][n channel][n dim]      value transform U_V, transposed
};
constexpr int MAX_GROUP_HEADS = 8;      // kv-heads per head group
constexpr int MAX_GROUP_QUERIES = 16;   // query heads per head-group stream (the decode's M tile)

struct Plan {
  uint32_t magic = PLAN_MAGIC;
  aatc_dims_t dims{};
  int n_streams = 0;
  int n_words = 0;        // W, words per record (plan-wide)
  int n_entries = 0;      // entries per stream in `entry` (32 * W)
  int max_bits = 0;       // widest channel of any stream
  int num_sms = 0;
  int device = 0;
  std::vector<int> retained;
  std::vector<int> nbits;
  std::vector<StreamLayout> layout;
  PlanDevice dev{};
  void* block = nullptr;  // single device allocation holding every table
  size_t block_bytes = 0;
  alignas(64) unsigned char tmap_u[128];   // CUtensorMap over ubf16_t (2D: 128 dims x S*128 rows)
  bool tmap_ok = false;
  int group_heads = 1;    // g_h: 1 for per-kv-head plans
  GroupDevice gdev{};
  alignas(64) unsigned char tmap_g[128];   // group plans: CUtensorMap over gdev.ubf (n dims x rows)
};

// Shape check shared by the planner (widths up to AATC_MAX_PLAN_BITS) and plan creation, which
// also rejects b_max > AATC_MAX_BITS as unsupported.
inline bool valid_dims(const aatc_dims_t* d) {
  return d && d->d == D && d->n_layers >= 1 && d->n_kv_heads >= 1 && d->n_q_heads >= d->n_kv_heads &&
         d->n_q_heads % d->n_kv_heads == 0 && d->b_max >= 1 && d->b_max <= AATC_MAX_PLAN_BITS &&
         d->n_layers <= 4096 && d->n_q_heads <= 4096;
}

struct CacheGeom {
  int n_tiles;
  size_t words_elems;     // uint32 elements of the word region
  size_t alpha_elems;     // fp32 elements of the alpha region
  size_t bytes;
};

inline CacheGeom cache_geom(int batch, int n_kv, int max_tokens, int n_words) {
  CacheGeom g;
  g.n_tiles = static_cast<int>((static_cast<int64_t>(max_tokens) + TILE - 1) / TILE);   // no int overflow
  g.words_elems = static_cast<size_t>(batch) * n_kv * 2 * g.n_tiles * n_words * TILE;
  g.alpha_elems = static_cast<size_t>(batch) * n_kv * 2 * g.n_tiles * TILE;
  g.bytes = 4 * (g.words_elems + g.alpha_elems);
  return g;
}

struct DecodeSplit {
  int n_splits;           // splits per (sequence, kv-head); split s covers tiles [s T / n, (s+1) T / n)
  int split_len;          // tokens of the longest split, a multiple of TILE
};

DecodeSplit decode_split(int batch, int n_kv, int n_ctx, int num_sms, int ctas_per_sm = 5);
// Split plan of the bf16 reference decode: the most CTAs per SM (up to 4) its shared memory
// allows, in one wave.
DecodeSplit bf16_decode_split(int batch, int n_kv, int n_q, int n_ctx, int num_sms);
// Dynamic shared memory of one bf16 reference split CTA (query columns padded to gp = 4 or 8).
size_t bf16_split_smem(int gp, int split_len);
// Decode workspace: split partials per (sequence, query head, split) -- 128 channel sums, then
// m, l, padded to a multiple of 4 floats -- followed by the per-call score A fragments per
// (sequence, kv-head) (up to 2 W k-steps x 32 lanes x 16 B), their offset corrections and score
// scales.
struct DecodeWs {
  int pstride;            // floats per partial
  int ks_stride;          // uint4 per (sequence, kv-head) fragment block
  size_t qfrag_off, qcorr_off, bytes;
};
DecodeWs decode_ws_layout(int batch, int n_q, int n_kv, int n_entries, int n_words, const DecodeSplit& sp);
size_t decode_workspace(int batch, int n_q, int n_kv, int n_entries, int n_words, const DecodeSplit& sp);
// The decode has two launch plans: the fused kernel (query rotation and split streaming in CTAs of
// 8-16 warps, FUSED_CTAS_PER_SM per SM, one wave) then the merge kernel, for layers whose streams
// share one of the record shapes it is built for; the query, split and merge kernels (about 5 CTAs
// per SM, at most 16 tiles per split) for any other layer.  `range` = the packed tokens a call covers, counted from the first tile it reads.
constexpr int FUSED_CTAS_PER_SM = 1;
DecodeSplit decode_split_for(int batch, int n_kv, int range, int num_sms, bool fused);
// Workspace bytes that serve a decode of `range` tokens on any layer of the plan, whichever path
// it takes.
size_t decode_workspace_for(const Plan& plan, int batch, int range);
// bf16 reference decode partials: 128 sums, then m, l, padding
size_t bf16_decode_workspace(int batch, int n_q, const DecodeSplit& sp);

// Handle check and CUDA-status mapping shared by every C entry point (defined in capi.cpp).
Plan* plan_from_handle(aatc_plan_t p);
aatc_status_t status_from_cuda(cudaError_t e);

// Raise `kernel`'s dynamic shared-memory limit on the current device to at least `bytes`.  The
// attribute belongs to a (device, kernel) pair, so what has been set is recorded per device and
// kernel under one mutex: host threads making first calls at the same time, and a process that
// drives several GPUs, both get the opt-in on every device they launch on (defined in capi.cpp).
cudaError_t ensure_smem_optin(const void* kernel, size_t bytes);

// Kernel launchers (defined in the .cu files); return the CUDA error of the launch.
// 2D tiled tensor map with 128-byte swizzle (16-bit elements): `map` is a 128-byte, 64-aligned
// CUtensorMap; rows of `inner` elements, `row_bytes` apart; box box_inner x box_rows.
cudaError_t make_tensor_map_2d(void* map, bool f16, const void* base, uint64_t inner, uint64_t rows,
                               uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows);
cudaError_t encode_tensor_maps_u(Plan& plan);
cudaError_t launch_encode(const Plan& plan, int layer, const void* K, const void* V, int batch,
                          int start, int n_tokens, void* cache, int max_tokens, cudaStream_t st);
// x: bf16 [batch][n_tokens][d_model] hidden states; a_hat: bf16 [L][H][2][128][d_model].
cudaError_t launch_encode_hidden(const Plan& plan, int layer, const void* x, int d_model, const void* a_hat,
                                 int batch, int start, int n_tokens, void* cache, int max_tokens, cudaStream_t st);
// Optional parts of a decode call: the packed range starts at token t_first (default 0), and
// n_full uncompressed tokens (bf16 [batch][full_cap][n_kv][128], e.g. a full-precision sink and
// recent window) join the same softmax.
struct DecodeExtra {
  int t_first = 0;
  const void* k_full = nullptr;
  const void* v_full = nullptr;
  int n_full = 0;
  int full_cap = 0;
};
constexpr int MAX_FULL_TOKENS = 8192;   // shared-memory scores of the uncompressed tokens
cudaError_t launch_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch,
                          int n_ctx, int max_tokens, float* out, void* ws, cudaStream_t st,
                          const DecodeExtra& extra);
// Prefill attention: codes workspace bytes, and the two launches (codes, attention).
size_t prefill_workspace(int batch, int n_kv, int n_ctx);
// The codes launch alone: the signed codes of every slot of `layer` for tokens [0, n_ctx) as f16
// in the prefill workspace layout ([b][slot][K|V][n_ctx_pad][128], value tiles transposed).
cudaError_t launch_codes(const Plan& plan, int layer, const void* cache, int batch, int n_ctx, int max_tokens,
                         void* ws, cudaStream_t st);
cudaError_t launch_prefill(const Plan& plan, int layer, const void* q, int q_start, int n_q, const void* cache,
                           int batch, int n_ctx, int max_tokens, float* out, void* ws, cudaStream_t st);
cudaError_t launch_dequant(const Plan& plan, int layer, const void* cache, int batch, int t0, int n,
                           int max_tokens, float* out, cudaStream_t st);
// Head-group plans (group.cu): encode of every group stream of a layer; decode workspace and
// launches (codes of the slices, folded queries, split attention, merge).
cudaError_t launch_group_encode(const Plan& plan, int layer, const void* K, const void* V, int batch, int start,
                                int n_tokens, void* cache, int max_tokens, cudaStream_t st);
size_t group_decode_workspace(const Plan& plan, int batch, int n_ctx);
cudaError_t launch_group_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                                int max_tokens, float* out, void* ws, cudaStream_t st);
cudaError_t launch_bf16_decode(const void* K, const void* V, const void* q, int batch, int n_ctx,
                               int max_tokens, int n_kv, int n_q, float* out, void* ws,
                               const DecodeSplit& sp, cudaStream_t st);

}  // namespace aatc
