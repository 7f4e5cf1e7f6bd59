// C ABI of the AATC library: argument validation, plan construction (packed-layout
// descriptor and per-channel constants) and dispatch to the CUDA kernels.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <utility>
#include <vector>

#include "aatc.h"
#include "aatc_internal.h"

namespace {

thread_local int32_t g_last_cuda_error = 0;

aatc_status_t cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return AATC_OK;
  g_last_cuda_error = static_cast<int32_t>(e);
  // the launchers answer cudaErrorNotSupported, before any launch, for a shape their kernels do
  // not implement (record tables beyond one SM's shared memory, more value tiles than a warp holds)
  return e == cudaErrorNotSupported ? AATC_ERR_UNSUPPORTED : AATC_ERR_CUDA;
}

aatc::Plan* as_plan(aatc_plan_t p) {
  auto* plan = reinterpret_cast<aatc::Plan*>(p);
  if (!plan || plan->magic != aatc::PLAN_MAGIC) return nullptr;
  return plan;
}

// fp32 -> bf16 bits, round to nearest even (inputs are finite; validated by the caller).
uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  const uint32_t round = 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>((u + round) >> 16);
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace aatc {

DecodeSplit decode_split(int batch, int n_kv, int n_ctx, int num_sms, int ctas_per_sm) {
  // About ctas_per_sm CTAs per SM in a single wave: n_splits per (sequence, kv-head), with split
  // s covering tiles [s T / n_splits, (s + 1) T / n_splits) so split lengths differ by at most
  // one tile and every SM gets nearly the same number of tiles.  A split holds at most 16 tiles
  // (its scores are kept in shared memory).
  const long tiles = (static_cast<long>(n_ctx) + TILE - 1) / TILE;
  const long units = static_cast<long>(batch) * n_kv;
  const long target = static_cast<long>(std::max(1, ctas_per_sm)) * std::max(1, num_sms);
  long n = (target + units / 2) / units;
  n = std::max(n, (tiles + 15) / 16);
  n = std::max(1L, std::min(n, tiles));
  DecodeSplit sp;
  sp.n_splits = static_cast<int>(n);
  sp.split_len = static_cast<int>((tiles + n - 1) / n) * TILE;   // longest split
  return sp;
}

DecodeSplit bf16_decode_split(int batch, int n_kv, int n_q, int n_ctx, int num_sms) {
  const int gp = n_q / n_kv <= 4 ? 4 : 8;
  constexpr size_t kSmPerSm = 228 * 1024, kReserved = 1024;   // per SM; reserved per CTA
  for (int c = 4; c > 1; --c) {
    const DecodeSplit sp = decode_split(batch, n_kv, n_ctx, num_sms, c);
    if (static_cast<size_t>(c) * (bf16_split_smem(gp, sp.split_len) + kReserved) <= kSmPerSm) return sp;
  }
  return decode_split(batch, n_kv, n_ctx, num_sms, 1);
}

Plan* plan_from_handle(aatc_plan_t p) { return as_plan(p); }

aatc_status_t status_from_cuda(cudaError_t e) { return cuda_status(e); }

cudaError_t ensure_smem_optin(const void* kernel, size_t bytes) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, size_t> done;   // (device, kernel) -> bytes set
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  size_t& have = done[std::make_pair(dev, kernel)];
  if (bytes <= have) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
  if (e == cudaSuccess) have = bytes;
  return e;
}

DecodeWs decode_ws_layout(int batch, int n_q, int n_kv, int n_entries, int n_words, const DecodeSplit& sp) {
  DecodeWs w;
  w.pstride = D + 4;                              // o_c per channel, then m, l (padded)
  w.ks_stride = 2 * n_words * 32;                 // >= score k16-steps (<= 2 W) x 32 lanes
  w.qfrag_off = align_up(static_cast<size_t>(batch) * n_q * sp.n_splits * w.pstride * sizeof(float), 256);
  w.qcorr_off = align_up(w.qfrag_off + static_cast<size_t>(batch) * n_kv * w.ks_stride * 16, 256);
  w.bytes = w.qcorr_off + static_cast<size_t>(batch) * n_kv * 2 * MAX_GROUP * sizeof(float);
  return w;
}

DecodeSplit decode_split_for(int batch, int n_kv, int range, int num_sms, bool fused) {
  if (!fused) return decode_split(batch, n_kv, std::max(range, 1), num_sms, 5);
  // fused kernel: one wave of at most FUSED_CTAS_PER_SM CTAs per SM; split lengths are not
  // bounded (the online softmax keeps no per-token scores)
  const long tiles = (static_cast<long>(std::max(range, 1)) + TILE - 1) / TILE;
  const long units = static_cast<long>(batch) * n_kv;
  long n = static_cast<long>(FUSED_CTAS_PER_SM) * std::max(1, num_sms) / units;
  n = std::max(1L, std::min(n, tiles));
  DecodeSplit sp;
  sp.n_splits = static_cast<int>(n);
  sp.split_len = static_cast<int>((tiles + n - 1) / n) * TILE;
  return sp;
}

size_t decode_workspace_for(const Plan& plan, int batch, int range) {
  const int hq = plan.dims.n_q_heads, hk = plan.dims.n_kv_heads;
  return std::max(decode_workspace(batch, hq, hk, plan.n_entries, plan.n_words,
                                   decode_split_for(batch, hk, range, plan.num_sms, false)),
                  decode_workspace(batch, hq, hk, plan.n_entries, plan.n_words,
                                   decode_split_for(batch, hk, range, plan.num_sms, true)));
}

size_t decode_workspace(int batch, int n_q, int n_kv, int n_entries, int n_words, const DecodeSplit& sp) {
  return decode_ws_layout(batch, n_q, n_kv, n_entries, n_words, sp).bytes;
}

size_t bf16_decode_workspace(int batch, int n_q, const DecodeSplit& sp) {
  return static_cast<size_t>(batch) * n_q * sp.n_splits * (D + 3) * sizeof(float);
}

// D2 / D1 record layout of one stream from its (non-increasing) widths; see StreamLayout.
void build_layout(const uint8_t* bits, StreamLayout* lay, std::vector<short>& entries) {
  std::vector<short> d2, d1;
  auto ent = [](int c, int sh) { return static_cast<short>(c | (sh << 8)); };
  for (int k = 0; k < 8; ++k) {
    int n = 0;
    for (int c = 0; c < D; ++c)
      if (bits[c] >= 2 * k + 2) {
        d2.push_back(ent(c, 2 * k));
        ++n;
      }
    lay->l2[k] = n;
    lay->l2all[k] = n;
    int m = 0;
    for (int c = 0; c < D; ++c) m += bits[c] >= 2 * k + 1;
    lay->lodd[k] = m;
  }
  for (int c = 0; c < D; ++c)
    if (bits[c] & 1) d1.push_back(ent(c, bits[c] - 1));
  const int r = static_cast<int>(d2.size()) % 16;
  for (int i = static_cast<int>(d2.size()) - r; i < static_cast<int>(d2.size()); ++i) {
    const int c = d2[i] & 0xFF, sh = d2[i] >> 8;
    d1.push_back(ent(c, sh));
    d1.push_back(ent(c, sh + 1));
  }
  d2.resize(d2.size() - r);
  for (int k = 7, left = r; k >= 0 && left > 0; --k) {      // the moved digits came off the last layers
    const int take = std::min(left, lay->l2[k]);
    lay->l2[k] -= take;
    left -= take;
  }
  lay->n2 = static_cast<int>(d2.size());
  lay->n1 = static_cast<int>(d1.size());
  lay->words = lay->n2 / 16 + (lay->n1 + 31) / 32;
  entries = d2;
  entries.insert(entries.end(), d1.begin(), d1.end());
}

}  // namespace aatc

extern "C" {

const char* aatc_status_string(aatc_status_t s) {
  switch (s) {
    case AATC_OK: return "ok";
    case AATC_ERR_INVALID_ARG: return "invalid argument";
    case AATC_ERR_BUDGET: return "bit budget not representable";
    case AATC_ERR_CAPACITY: return "token range exceeds cache capacity";
    case AATC_ERR_WORKSPACE: return "workspace too small";
    case AATC_ERR_UNSUPPORTED: return "unsupported shape";
    case AATC_ERR_CUDA: return "CUDA error";
    case AATC_ERR_NOMEM: return "out of memory";
    case AATC_ERR_DEVICE_FLAG: return "device error flag set";
    case AATC_ERR_IO: return "plan file unreadable or corrupt";
  }
  return "unknown status";
}

int32_t aatc_last_cuda_error(void) { return g_last_cuda_error; }

int32_t aatc_version(void) { return 200; }   // 0.2.0: plan files, AATC_ERR_IO, planner widths to 16

namespace {

// Device plan from per-slot widths and scales ([L][H_kv][2][128]).  Per-kv-head plans pass the
// per-slot bases (g_h = 1); head-group plans pass g_h > 1, no per-slot basis, and the group bases
// gbasis [L][H_kv / g_h][2][n][n] (dim x storage channel, n = 128 g_h) whose slices the slots hold.
aatc_status_t create_plan(const aatc_dims_t* dims, const float* basis, const uint8_t* bits, const float* scales,
                          int g_h, const float* gbasis, void* stream, aatc_plan_t* plan_out) {
  using namespace aatc;
  if (!valid_dims(dims) || (!basis && !gbasis) || !bits || !scales || !plan_out) return AATC_ERR_INVALID_ARG;
  if (dims->b_max > AATC_MAX_BITS) return AATC_ERR_UNSUPPORTED;
  const int S = dims->n_layers * dims->n_kv_heads * 2;
  const size_t SD = static_cast<size_t>(S) * D;
  // validate
  std::vector<int> retained(S), nbits(S);
  for (int s = 0; s < S; ++s) {
    int r = 0, nb = 0;
    for (int c = 0; c < D; ++c) {
      const int b = bits[s * D + c];
      if (b > dims->b_max) return AATC_ERR_INVALID_ARG;
      if (c > 0 && b > bits[s * D + c - 1]) return AATC_ERR_INVALID_ARG;   // non-increasing
      if (b > 8 && c >= kMaxWideChannels) return AATC_ERR_UNSUPPORTED;
      if (b > 0) {
        const float sc = scales[s * D + c];
        if (!(std::isfinite(sc) && sc > 0.0f)) return AATC_ERR_INVALID_ARG;
        ++r;
      }
      nb += b;
    }
    retained[s] = r;
    nbits[s] = nb;
  }
  const int n_g = D * g_h, NG = dims->n_kv_heads / g_h;
  const size_t GB = static_cast<size_t>(dims->n_layers) * NG * 2 * n_g * n_g;   // group basis elements
  if (basis) {
    for (size_t i = 0; i < SD * D; ++i)
      if (!std::isfinite(basis[i])) return AATC_ERR_INVALID_ARG;
  } else {
    for (size_t i = 0; i < GB; ++i)
      if (!std::isfinite(gbasis[i])) return AATC_ERR_INVALID_ARG;
  }
  std::vector<StreamLayout> layout(S);
  std::vector<std::vector<short>> entries(S);
  int W = 1;
  for (int s = 0; s < S; ++s) {
    build_layout(bits + static_cast<size_t>(s) * D, &layout[s], entries[s]);
    layout[s].nret = retained[s];
    W = std::max(W, layout[s].words);
  }
  const int E = 32 * W;                                             // entries per stream (padded)

  // host staging of every table, in one block
  size_t off = 0;
  const size_t SDD = basis ? SD * D : 0;                            // per-slot basis tables
  const size_t GBk = basis ? 0 : GB;                                // group tables
  const size_t o_ubf = off;  off = align_up(off + SDD * 2, 256);
  const size_t o_u32 = off;  off = align_up(off + SDD * 4, 256);
  const size_t o_u32t = off; off = align_up(off + SDD * 4, 256);
  const size_t o_gubf = off; off = align_up(off + GBk * 2, 256);
  const size_t o_guk = off;  off = align_up(off + GBk / 2 * 4, 256);
  const size_t o_guvt = off; off = align_up(off + GBk / 2 * 4, 256);
  const size_t o_enc = off;  off = align_up(off + SD * sizeof(ChanEnc), 256);
  const size_t o_invs = off; off = align_up(off + SD * 4, 256);
  const size_t o_f = off;    off = align_up(off + SD * 4, 256);
  const size_t o_lay = off;  off = align_up(off + static_cast<size_t>(S) * sizeof(StreamLayout), 256);
  const size_t o_ent = off;  off = align_up(off + static_cast<size_t>(S) * E * sizeof(short), 256);
  const size_t o_che = off;  off = align_up(off + SD * kChanEnt * sizeof(short), 256);
  const size_t o_err = off;  off = align_up(off + 16, 256);
  const size_t total = off;
  std::vector<unsigned char> host;
  try {
    host.assign(total, 0);
  } catch (const std::bad_alloc&) {
    return AATC_ERR_NOMEM;
  }
  auto* ubf = reinterpret_cast<uint16_t*>(host.data() + o_ubf);
  auto* u32 = reinterpret_cast<float*>(host.data() + o_u32);
  auto* u32t = reinterpret_cast<float*>(host.data() + o_u32t);
  auto* enc = reinterpret_cast<ChanEnc*>(host.data() + o_enc);
  auto* invs = reinterpret_cast<float*>(host.data() + o_invs);
  auto* fc = reinterpret_cast<float*>(host.data() + o_f);
  auto* lay = reinterpret_cast<StreamLayout*>(host.data() + o_lay);
  auto* ent = reinterpret_cast<short*>(host.data() + o_ent);
  auto* che = reinterpret_cast<short*>(host.data() + o_che);
  if (!basis) {
    // group tables, channels in slice-major order: j' = 128 s + c holds storage channel c g_h + s
    auto* gubf = reinterpret_cast<uint16_t*>(host.data() + o_gubf);
    auto* guk = reinterpret_cast<float*>(host.data() + o_guk);
    auto* guvt = reinterpret_cast<float*>(host.data() + o_guvt);
    const size_t nn = static_cast<size_t>(n_g) * n_g;
    for (int l = 0; l < dims->n_layers; ++l)
      for (int g = 0; g < NG; ++g)
        for (int kind = 0; kind < 2; ++kind) {
          const size_t sg = (static_cast<size_t>(l) * NG + g) * 2 + kind;
          const float* ub = gbasis + sg * nn;                       // [dim][storage channel]
          for (int jp = 0; jp < n_g; ++jp) {
            const int j = (jp % D) * g_h + jp / D;
            for (int d = 0; d < n_g; ++d) {
              const float v = ub[static_cast<size_t>(d) * n_g + j];
              gubf[sg * nn + static_cast<size_t>(jp) * n_g + d] = f32_to_bf16_rne(v);
              const size_t lg = (static_cast<size_t>(l) * NG + g) * nn;
              if (kind == 0) guk[lg + static_cast<size_t>(d) * n_g + jp] = v;
              else guvt[lg + static_cast<size_t>(jp) * n_g + d] = v;
            }
          }
        }
  }
  for (int s = 0; s < S; ++s) {
    if (basis) {
      const float* bs = basis + static_cast<size_t>(s) * D * D;   // [dim][channel]
      for (int d = 0; d < D; ++d)
        for (int c = 0; c < D; ++c) {
          ubf[(static_cast<size_t>(s) * D + c) * D + d] = f32_to_bf16_rne(bs[d * D + c]);
          u32[(static_cast<size_t>(s) * D + d) * D + c] = bs[d * D + c];
          u32t[(static_cast<size_t>(s) * D + c) * D + d] = bs[d * D + c];
        }
    }
    for (int c = 0; c < D; ++c) {
      const size_t i = static_cast<size_t>(s) * D + c;
      const int b = bits[i];
      ChanEnc e{0.0f, 0.0f, 12582912.0f, 0.0f};
      if (b > 0) {
        const float f = std::ldexp(scales[i], 1 - b);            // exact power-of-two scaling
        e.inv_f = 1.0f / f;
        e.hi = std::ldexp(1.0f, b - 1) - 1.0f;
        e.magic = 12582912.0f + std::ldexp(1.0f, b - 1);
        e.off = std::ldexp(1.0f, b - 1);
        fc[i] = f;
        invs[i] = 1.0f / scales[i];
      }
      enc[i] = e;
    }
    lay[s] = layout[s];
    for (int e = 0; e < E; ++e)
      ent[static_cast<size_t>(s) * E + e] = e < static_cast<int>(entries[s].size()) ? entries[s][e] : short(-1);
    short* ce = che + static_cast<size_t>(s) * D * kChanEnt;
    for (int i = 0; i < D * kChanEnt; ++i) ce[i] = -1;
    int fill[D] = {0};
    for (int e = 0; e < static_cast<int>(entries[s].size()); ++e) {
      const int c = entries[s][e] & 0xFF;
      if (fill[c] < kChanEnt) ce[c * kChanEnt + fill[c]++] = static_cast<short>(e);
    }
  }

  auto* plan = new (std::nothrow) Plan();
  if (!plan) return AATC_ERR_NOMEM;
  plan->dims = *dims;
  plan->n_streams = S;
  plan->n_words = W;
  plan->n_entries = E;
  for (size_t i = 0; i < SD; ++i) plan->max_bits = std::max(plan->max_bits, static_cast<int>(bits[i]));
  plan->retained = retained;
  plan->nbits = nbits;
  plan->layout = layout;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaGetDevice(&plan->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&plan->num_sms, cudaDevAttrMultiProcessorCount, plan->device);
  if (e == cudaSuccess) e = cudaMalloc(&plan->block, total);
  if (e != cudaSuccess) {
    delete plan;
    return e == cudaErrorMemoryAllocation ? AATC_ERR_NOMEM : cuda_status(e);
  }
  plan->block_bytes = total;
  e = cudaMemcpyAsync(plan->block, host.data(), total, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  auto* base = static_cast<unsigned char*>(plan->block);
  plan->dev.ubf16_t = base + o_ubf;
  plan->dev.u32 = reinterpret_cast<const float*>(base + o_u32);
  plan->dev.u32t = reinterpret_cast<const float*>(base + o_u32t);
  plan->dev.enc = reinterpret_cast<const ChanEnc*>(base + o_enc);
  plan->dev.inv_s = reinterpret_cast<const float*>(base + o_invs);
  plan->dev.f = reinterpret_cast<const float*>(base + o_f);
  plan->dev.lay = reinterpret_cast<const StreamLayout*>(base + o_lay);
  plan->dev.entry = reinterpret_cast<const short*>(base + o_ent);
  plan->dev.chan_ent = reinterpret_cast<const short*>(base + o_che);
  plan->dev.err = reinterpret_cast<int*>(base + o_err);
  plan->group_heads = g_h;
  if (basis) {
    if (e == cudaSuccess) e = encode_tensor_maps_u(*plan);
  } else {
    plan->dev.ubf16_t = nullptr;
    plan->dev.u32 = plan->dev.u32t = nullptr;
    plan->gdev.ubf = base + o_gubf;
    plan->gdev.uk = reinterpret_cast<const float*>(base + o_guk);
    plan->gdev.uvt = reinterpret_cast<const float*>(base + o_guvt);
    // rows of n_g dims, one per (layer, group, kind, slice-major channel); box 64 dims x 256 rows
    if (e == cudaSuccess)
      e = make_tensor_map_2d(plan->tmap_g, false, plan->gdev.ubf, static_cast<uint64_t>(n_g), GB / n_g,
                             static_cast<uint64_t>(n_g) * 2, 64, 256);
  }
  if (e != cudaSuccess) {
    cudaFree(plan->block);
    delete plan;
    return cuda_status(e);
  }
  *plan_out = reinterpret_cast<aatc_plan_t>(plan);
  return AATC_OK;
}

}  // namespace

aatc_status_t aatc_plan_create(const aatc_dims_t* dims, const float* basis, const uint8_t* bits,
                               const float* scales, void* stream, aatc_plan_t* plan_out) {
  if (!basis) return AATC_ERR_INVALID_ARG;
  return create_plan(dims, basis, bits, scales, 1, nullptr, stream, plan_out);
}

aatc_status_t aatc_group_plan_create(const aatc_dims_t* dims, int32_t g_h, const float* basis, const uint8_t* bits,
                                     const float* scales, void* stream, aatc_plan_t* plan_out) {
  using namespace aatc;
  if (!valid_dims(dims) || !basis || !bits || !scales || !plan_out || g_h < 2 || g_h > MAX_GROUP_HEADS ||
      dims->n_kv_heads % g_h != 0)
    return AATC_ERR_INVALID_ARG;
  if (dims->b_max > 8 || (g_h != 2 && g_h != 4) || (dims->n_q_heads / dims->n_kv_heads) * g_h > MAX_GROUP_QUERIES)
    return AATC_ERR_UNSUPPORTED;                    // TMEM holds the 128 g_h channels of a token tile: g_h <= 4
  const int n = D * g_h, NG = dims->n_kv_heads / g_h, L = dims->n_layers;
  // the slots' slices: slot (l, g g_h + s, kind) channel c = storage channel c g_h + s
  const size_t S = static_cast<size_t>(L) * dims->n_kv_heads * 2;
  std::vector<uint8_t> sb(S * D);
  std::vector<float> ss(S * D);
  for (int l = 0; l < L; ++l)
    for (int g = 0; g < NG; ++g)
      for (int kind = 0; kind < 2; ++kind) {
        const size_t sg = (static_cast<size_t>(l) * NG + g) * 2 + kind;
        const uint8_t* gb = bits + sg * n;
        const float* gs = scales + sg * n;
        for (int j = 0; j < n; ++j) {
          if (gb[j] > dims->b_max || (j > 0 && gb[j] > gb[j - 1])) return AATC_ERR_INVALID_ARG;
          if (gb[j] > 0 && !(std::isfinite(gs[j]) && gs[j] > 0.0f)) return AATC_ERR_INVALID_ARG;
          const int sl = j % g_h, c = j / g_h;
          const size_t slot = (static_cast<size_t>(l) * dims->n_kv_heads + g * g_h + sl) * 2 + kind;
          sb[slot * D + c] = gb[j];
          ss[slot * D + c] = gs[j];
        }
      }
  return create_plan(dims, nullptr, sb.data(), ss.data(), g_h, basis, stream, plan_out);
}

aatc_status_t aatc_plan_destroy(aatc_plan_t p) {
  if (!p) return AATC_OK;
  aatc::Plan* plan = as_plan(p);
  if (!plan) return AATC_ERR_INVALID_ARG;
  cudaError_t e = cudaDeviceSynchronize();
  cudaError_t e2 = cudaFree(plan->block);
  plan->magic = aatc::PLAN_DEAD;
  delete plan;
  if (e != cudaSuccess) return cuda_status(e);
  return cuda_status(e2);
}

aatc_status_t aatc_plan_info(aatc_plan_t p, int32_t* n_words, int32_t* retained) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !n_words) return AATC_ERR_INVALID_ARG;
  *n_words = plan->n_words;
  if (retained)
    for (int s = 0; s < plan->n_streams; ++s) retained[s] = plan->retained[s];
  return AATC_OK;
}

aatc_status_t aatc_cache_bytes(aatc_plan_t p, int32_t batch, int32_t max_tokens, size_t* bytes) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !bytes || batch < 1 || max_tokens < 1) return AATC_ERR_INVALID_ARG;
  *bytes = aatc::cache_geom(batch, plan->dims.n_kv_heads, max_tokens, plan->n_words).bytes;
  return AATC_OK;
}

aatc_status_t aatc_encode(aatc_plan_t p, int32_t layer, const void* K, const void* V, int32_t batch,
                          int32_t start, int32_t n_tokens, void* cache, int32_t max_tokens,
                          void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || layer < 0 || layer >= plan->dims.n_layers || batch < 1 || start < 0 || n_tokens < 0 ||
      max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (static_cast<int64_t>(start) + n_tokens > max_tokens) return AATC_ERR_CAPACITY;
  if (n_tokens == 0) return AATC_OK;                   // an empty append reads no pointer
  if (!K || !V || !cache || !aligned16(K) || !aligned16(V) || !aligned16(cache)) return AATC_ERR_INVALID_ARG;
  if (plan->group_heads > 1)
    return cuda_status(aatc::launch_group_encode(*plan, layer, K, V, batch, start, n_tokens, cache, max_tokens,
                                                 static_cast<cudaStream_t>(stream)));
  return cuda_status(aatc::launch_encode(*plan, layer, K, V, batch, start, n_tokens, cache,
                                         max_tokens, static_cast<cudaStream_t>(stream)));
}

aatc_status_t aatc_encode_hidden(aatc_plan_t p, int32_t layer, const void* x, int32_t d_model, const void* a_hat,
                                 int32_t batch, int32_t start, int32_t n_tokens, void* cache, int32_t max_tokens,
                                 void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || layer < 0 || layer >= plan->dims.n_layers || batch < 1 || start < 0 || n_tokens < 0 ||
      max_tokens < 1 || d_model < 64 || d_model % 64 != 0 || d_model > 65536)
    return AATC_ERR_INVALID_ARG;
  if (static_cast<int64_t>(start) + n_tokens > max_tokens) return AATC_ERR_CAPACITY;
  if (n_tokens == 0) return AATC_OK;                   // an empty append reads no pointer
  if (!x || !a_hat || !cache || !aligned16(x) || !aligned16(a_hat) || !aligned16(cache))
    return AATC_ERR_INVALID_ARG;
  if (plan->max_bits > 8 || plan->group_heads > 1) return AATC_ERR_UNSUPPORTED;   // one byte per stored value; per-kv-head slots
  return cuda_status(aatc::launch_encode_hidden(*plan, layer, x, d_model, a_hat, batch, start, n_tokens, cache,
                                                max_tokens, static_cast<cudaStream_t>(stream)));
}

aatc_status_t aatc_prefill_workspace_bytes(aatc_plan_t p, int32_t batch, int32_t n_ctx, size_t* bytes) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !bytes || batch < 1 || n_ctx < 1) return AATC_ERR_INVALID_ARG;
  *bytes = aatc::prefill_workspace(batch, plan->dims.n_kv_heads, n_ctx);
  return AATC_OK;
}

aatc_status_t aatc_prefill_attention(aatc_plan_t p, int32_t layer, const void* q, int32_t q_start, int32_t n_q,
                                     const void* cache, int32_t batch, int32_t n_ctx, int32_t max_tokens, float* out,
                                     void* workspace, size_t workspace_bytes, void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !q || !cache || !out || !workspace || layer < 0 || layer >= plan->dims.n_layers || batch < 1 ||
      q_start < 0 || n_q < 1 || n_ctx < 1 || max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (n_ctx > max_tokens) return AATC_ERR_CAPACITY;
  if (static_cast<int64_t>(q_start) + n_q > n_ctx) return AATC_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(cache) || !aligned16(out) || !aligned16(workspace)) return AATC_ERR_INVALID_ARG;
  if (plan->n_words > 32) return AATC_ERR_UNSUPPORTED;
  if (plan->max_bits > 12) return AATC_ERR_UNSUPPORTED;   // f16 code operands are exact up to |code| = 2048
  if (plan->group_heads > 1) return AATC_ERR_UNSUPPORTED;
  if (workspace_bytes < aatc::prefill_workspace(batch, plan->dims.n_kv_heads, n_ctx)) return AATC_ERR_WORKSPACE;
  return cuda_status(aatc::launch_prefill(*plan, layer, q, q_start, n_q, cache, batch, n_ctx, max_tokens, out,
                                          workspace, static_cast<cudaStream_t>(stream)));
}

aatc_status_t aatc_decode_workspace_bytes(aatc_plan_t p, int32_t batch, int32_t n_ctx, size_t* bytes) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !bytes || batch < 1 || n_ctx < 1) return AATC_ERR_INVALID_ARG;
  *bytes = plan->group_heads > 1 ? aatc::group_decode_workspace(*plan, batch, n_ctx)
                                 : aatc::decode_workspace_for(*plan, batch, n_ctx);
  return AATC_OK;
}

aatc_status_t aatc_decode_attention(aatc_plan_t p, int32_t layer, const void* q, const void* cache,
                                    int32_t batch, int32_t n_ctx, int32_t max_tokens, float* out,
                                    void* workspace, size_t workspace_bytes, void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !q || !cache || !out || !workspace || layer < 0 || layer >= plan->dims.n_layers ||
      batch < 1 || n_ctx < 1 || max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (n_ctx > max_tokens) return AATC_ERR_CAPACITY;
  if (plan->dims.n_q_heads / plan->dims.n_kv_heads > aatc::MAX_GROUP) return AATC_ERR_UNSUPPORTED;
  if (!aligned16(cache) || !aligned16(workspace)) return AATC_ERR_INVALID_ARG;
  if (plan->group_heads > 1) {
    if (!aligned16(q) || !aligned16(out)) return AATC_ERR_INVALID_ARG;
    if (workspace_bytes < aatc::group_decode_workspace(*plan, batch, n_ctx)) return AATC_ERR_WORKSPACE;
    return cuda_status(aatc::launch_group_decode(*plan, layer, q, cache, batch, n_ctx, max_tokens, out, workspace,
                                                 static_cast<cudaStream_t>(stream)));
  }
  if (workspace_bytes < aatc::decode_workspace_for(*plan, batch, n_ctx)) return AATC_ERR_WORKSPACE;
  return cuda_status(aatc::launch_decode(*plan, layer, q, cache, batch, n_ctx, max_tokens, out,
                                         workspace, static_cast<cudaStream_t>(stream), aatc::DecodeExtra{}));
}

aatc_status_t aatc_decode_attention_sw(aatc_plan_t p, int32_t layer, const void* q, const void* cache,
                                       int32_t batch, int32_t t_first, int32_t t_end, int32_t max_tokens,
                                       const void* k_full, const void* v_full, int32_t n_full, int32_t full_cap,
                                       float* out, void* workspace, size_t workspace_bytes, void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !q || !cache || !out || layer < 0 || layer >= plan->dims.n_layers || batch < 1 ||
      max_tokens < 1 || t_first < 0 || t_end < t_first || n_full < 0 || (n_full > 0 && (!k_full || !v_full)) ||
      full_cap < n_full || (t_end == t_first && n_full == 0))
    return AATC_ERR_INVALID_ARG;
  if (t_end > max_tokens || n_full > aatc::MAX_FULL_TOKENS) return AATC_ERR_CAPACITY;
  if (plan->dims.n_q_heads / plan->dims.n_kv_heads > aatc::MAX_GROUP || plan->group_heads > 1)
    return AATC_ERR_UNSUPPORTED;
  if (!aligned16(cache) || (n_full > 0 && (!aligned16(k_full) || !aligned16(v_full)))) return AATC_ERR_INVALID_ARG;
  // the packed part covers tiles [t_first / 128, ceil(t_end / 128)): never more splits than a
  // plain decode of t_end tokens, so aatc_decode_workspace_bytes(batch, t_end) suffices
  const int range = t_end - (t_first / aatc::TILE) * aatc::TILE;
  if (t_end > t_first) {
    if (!workspace || !aligned16(workspace)) return AATC_ERR_INVALID_ARG;
    if (workspace_bytes < aatc::decode_workspace_for(*plan, batch, range)) return AATC_ERR_WORKSPACE;
  }
  aatc::DecodeExtra ex;
  ex.t_first = t_first;
  ex.k_full = k_full;
  ex.v_full = v_full;
  ex.n_full = n_full;
  ex.full_cap = full_cap;
  return cuda_status(aatc::launch_decode(*plan, layer, q, cache, batch, t_end, max_tokens, out, workspace,
                                         static_cast<cudaStream_t>(stream), ex));
}

aatc_status_t aatc_dequantize(aatc_plan_t p, int32_t layer, const void* cache, int32_t batch,
                              int32_t t0, int32_t n, int32_t max_tokens, float* coeffs_out,
                              void* stream) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !cache || !coeffs_out || layer < 0 || layer >= plan->dims.n_layers || batch < 1 ||
      t0 < 0 || n < 0 || max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (static_cast<int64_t>(t0) + n > max_tokens) return AATC_ERR_CAPACITY;
  if (n == 0) return AATC_OK;
  return cuda_status(aatc::launch_dequant(*plan, layer, cache, batch, t0, n, max_tokens, coeffs_out,
                                          static_cast<cudaStream_t>(stream)));
}

aatc_status_t aatc_get_device_error(aatc_plan_t p, int32_t* flags, int32_t clear) {
  aatc::Plan* plan = as_plan(p);
  if (!plan || !flags) return AATC_ERR_INVALID_ARG;
  int32_t h[4] = {0, 0, 0, 0};
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(h, plan->dev.err, sizeof(h), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && clear) e = cudaMemset(plan->dev.err, 0, sizeof(h));
  if (e != cudaSuccess) return cuda_status(e);
  *flags = h[0];
  return AATC_OK;
}

aatc_status_t aatc_bf16_decode_workspace_bytes(int32_t batch, int32_t n_kv, int32_t n_q, int32_t n_ctx,
                                               size_t* bytes) {
  if (!bytes || batch < 1 || n_kv < 1 || n_q < n_kv || n_q % n_kv || n_ctx < 1) return AATC_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    sms = 1;
  *bytes = aatc::bf16_decode_workspace(batch, n_q, aatc::bf16_decode_split(batch, n_kv, n_q, n_ctx, sms));
  return AATC_OK;
}

aatc_status_t aatc_bf16_decode_attention(const void* K, const void* V, const void* q, int32_t batch,
                                         int32_t n_ctx, int32_t max_tokens, int32_t n_kv, int32_t n_q,
                                         float* out, void* workspace, size_t workspace_bytes,
                                         void* stream) {
  if (!K || !V || !q || !out || !workspace || batch < 1 || n_ctx < 1 || n_kv < 1 || n_q < n_kv ||
      n_q % n_kv || max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (n_ctx > max_tokens) return AATC_ERR_CAPACITY;
  if (n_q / n_kv > aatc::MAX_GROUP) return AATC_ERR_UNSUPPORTED;
  if (!aligned16(K) || !aligned16(V) || !aligned16(workspace)) return AATC_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_status(e);
  const auto sp = aatc::bf16_decode_split(batch, n_kv, n_q, n_ctx, sms);
  if (workspace_bytes < aatc::bf16_decode_workspace(batch, n_q, sp)) return AATC_ERR_WORKSPACE;
  return cuda_status(aatc::launch_bf16_decode(K, V, q, batch, n_ctx, max_tokens, n_kv, n_q, out,
                                              workspace, sp, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
