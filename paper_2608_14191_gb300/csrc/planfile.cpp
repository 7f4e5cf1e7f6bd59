// Plan files: the calibration outputs (basis, widths, scales) of Algorithm 1's offline half written
// once and read back, so a model is calibrated once and its plans are recreated from disk.
//
// Layout, every field little-endian whatever the host:
//   magic "AATCPLAN" (8 bytes), u32 version = 1, u32 header bytes = 48,
//   i32 d, n_layers, n_kv_heads, n_q_heads, b_max,  u32 reserved = 0,
//   u64 payload bytes,
//   payload: basis fp32 [S][128][128], bits u8 [S][128], scales fp32 [S][128]   (S = L * H_kv * 2),
//   u64 FNV-1a (64-bit) of the payload bytes.
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <vector>

#include "aatc_internal.h"

namespace {

constexpr char kMagic[8] = {'A', 'A', 'T', 'C', 'P', 'L', 'A', 'N'};
constexpr uint32_t kVersion = 1;
constexpr uint32_t kHeaderBytes = 48;

void put_u32(std::vector<unsigned char>& o, uint32_t v) {
  for (int i = 0; i < 4; ++i) o.push_back(static_cast<unsigned char>(v >> (8 * i)));
}
void put_u64(std::vector<unsigned char>& o, uint64_t v) {
  for (int i = 0; i < 8; ++i) o.push_back(static_cast<unsigned char>(v >> (8 * i)));
}
uint32_t get_u32(const unsigned char* p) {
  uint32_t v = 0;
  for (int i = 0; i < 4; ++i) v |= static_cast<uint32_t>(p[i]) << (8 * i);
  return v;
}
uint64_t get_u64(const unsigned char* p) {
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= static_cast<uint64_t>(p[i]) << (8 * i);
  return v;
}

uint64_t fnv1a64(const unsigned char* p, size_t n) {
  uint64_t h = 1469598103934665603ull;
  for (size_t i = 0; i < n; ++i) {
    h ^= p[i];
    h *= 1099511628211ull;
  }
  return h;
}

size_t n_streams(const aatc_dims_t& d) { return static_cast<size_t>(d.n_layers) * d.n_kv_heads * 2; }
size_t payload_bytes(const aatc_dims_t& d) {
  const size_t S = n_streams(d);
  return S * aatc::D * aatc::D * 4 + S * aatc::D + S * aatc::D * 4;
}

// Reads and checks a whole plan file: header, sizes and checksum.  On success `dims` and `payload`
// hold the file's contents.
aatc_status_t read_file(const char* path, aatc_dims_t* dims, std::vector<unsigned char>* payload) {
  std::FILE* f = std::fopen(path, "rb");
  if (!f) return AATC_ERR_IO;
  unsigned char hdr[kHeaderBytes];
  aatc_status_t st = AATC_OK;
  if (std::fread(hdr, 1, kHeaderBytes, f) != kHeaderBytes || std::memcmp(hdr, kMagic, 8) != 0 ||
      get_u32(hdr + 8) != kVersion || get_u32(hdr + 12) != kHeaderBytes) {
    st = AATC_ERR_IO;
  } else {
    aatc_dims_t d;
    d.d = static_cast<int32_t>(get_u32(hdr + 16));
    d.n_layers = static_cast<int32_t>(get_u32(hdr + 20));
    d.n_kv_heads = static_cast<int32_t>(get_u32(hdr + 24));
    d.n_q_heads = static_cast<int32_t>(get_u32(hdr + 28));
    d.b_max = static_cast<int32_t>(get_u32(hdr + 32));
    const uint64_t nbytes = get_u64(hdr + 40);
    if (!aatc::valid_dims(&d) || get_u32(hdr + 36) != 0 || nbytes != payload_bytes(d)) {
      st = AATC_ERR_IO;
    } else {
      payload->resize(static_cast<size_t>(nbytes));
      unsigned char tail[8];
      if (std::fread(payload->data(), 1, payload->size(), f) != payload->size() || std::fread(tail, 1, 8, f) != 8 ||
          std::fgetc(f) != EOF || get_u64(tail) != fnv1a64(payload->data(), payload->size())) {
        st = AATC_ERR_IO;                               // short, trailing bytes or checksum mismatch
      } else {
        const size_t S = n_streams(d);
        const unsigned char* bits = payload->data() + S * aatc::D * aatc::D * 4;
        for (size_t i = 0; i < S * aatc::D && st == AATC_OK; ++i)
          if (bits[i] > d.b_max) st = AATC_ERR_IO;
        if (st == AATC_OK) *dims = d;
      }
    }
  }
  std::fclose(f);
  return st;
}

}  // namespace

extern "C" aatc_status_t aatc_plan_save(const char* path, const aatc_dims_t* dims, const float* basis,
                                        const uint8_t* bits, const float* scales) {
  using namespace aatc;
  if (!path || !aatc::valid_dims(dims) || !basis || !bits || !scales) return AATC_ERR_INVALID_ARG;
  const size_t S = n_streams(*dims);
  for (size_t i = 0; i < S * D; ++i)
    if (bits[i] > dims->b_max) return AATC_ERR_INVALID_ARG;
  std::vector<unsigned char> out;
  out.reserve(kHeaderBytes + payload_bytes(*dims) + 8);
  out.insert(out.end(), kMagic, kMagic + 8);
  put_u32(out, kVersion);
  put_u32(out, kHeaderBytes);
  put_u32(out, static_cast<uint32_t>(dims->d));
  put_u32(out, static_cast<uint32_t>(dims->n_layers));
  put_u32(out, static_cast<uint32_t>(dims->n_kv_heads));
  put_u32(out, static_cast<uint32_t>(dims->n_q_heads));
  put_u32(out, static_cast<uint32_t>(dims->b_max));
  put_u32(out, 0);
  put_u64(out, payload_bytes(*dims));
  const size_t p0 = out.size();
  for (size_t i = 0; i < S * D * D; ++i) {
    uint32_t u;
    std::memcpy(&u, basis + i, 4);
    put_u32(out, u);
  }
  out.insert(out.end(), bits, bits + S * D);
  for (size_t i = 0; i < S * D; ++i) {
    uint32_t u;
    std::memcpy(&u, scales + i, 4);
    put_u32(out, u);
  }
  put_u64(out, fnv1a64(out.data() + p0, out.size() - p0));
  std::FILE* f = std::fopen(path, "wb");
  if (!f) return AATC_ERR_IO;
  const bool ok = std::fwrite(out.data(), 1, out.size(), f) == out.size();
  const bool closed = std::fclose(f) == 0;
  return ok && closed ? AATC_OK : AATC_ERR_IO;
}

extern "C" aatc_status_t aatc_plan_file_dims(const char* path, aatc_dims_t* dims_out) {
  if (!path || !dims_out) return AATC_ERR_INVALID_ARG;
  std::vector<unsigned char> payload;
  aatc_dims_t d;
  const aatc_status_t st = read_file(path, &d, &payload);
  if (st == AATC_OK) *dims_out = d;
  return st;
}

extern "C" aatc_status_t aatc_plan_load(const char* path, const aatc_dims_t* dims, float* basis_out,
                                        uint8_t* bits_out, float* scales_out) {
  using namespace aatc;
  if (!path || !dims || !basis_out || !bits_out || !scales_out) return AATC_ERR_INVALID_ARG;
  std::vector<unsigned char> payload;
  aatc_dims_t d;
  const aatc_status_t st = read_file(path, &d, &payload);
  if (st != AATC_OK) return st;
  if (d.d != dims->d || d.n_layers != dims->n_layers || d.n_kv_heads != dims->n_kv_heads ||
      d.n_q_heads != dims->n_q_heads || d.b_max != dims->b_max)
    return AATC_ERR_INVALID_ARG;
  const size_t S = n_streams(d);
  const unsigned char* p = payload.data();
  for (size_t i = 0; i < S * D * D; ++i, p += 4) {
    const uint32_t u = get_u32(p);
    std::memcpy(basis_out + i, &u, 4);
  }
  std::memcpy(bits_out, p, S * D);
  p += S * D;
  for (size_t i = 0; i < S * D; ++i, p += 4) {
    const uint32_t u = get_u32(p);
    std::memcpy(scales_out + i, &u, 4);
  }
  return AATC_OK;
}
