// Strict 5-bit code storage (Sec. 4: a weight is 4 shift bits and a sign
// bit).  With shifts in [-14, 0] a ternary sign times 15 shifts plus the zero
// weight is 31 states, which fit 5 bits: code 0 is the zero weight, 1 + (-p)
// a weight with s = +1, 16 + (-p) one with s = -1 (31 is never written).  The
// full [-15, 0] range needs the 6-bit planes of ds_pack_shift_weights; this
// format is storage only (compute calls take the 6-bit blob and its expanded
// layout), converted with ds_pack_shift_weights5 / ds_unpack_shift_weights5.
//
// Blob: a 256-byte header (u32 magic, u32 format = 2, i64 n_out, i64 k_red,
// i64 n_chunks, u32 invalid_count), then n_out x n_chunks records of 5 u32:
// word b of record (n, g) holds bit b of the code of k = 32 g + j at bit j.
// One warp packs one record: lane j forms the code of weight j and the five
// words are the warp's ballots of its bits.
#include <cstddef>
#include <mutex>

#include "ds_common.cuh"

namespace {

constexpr uint32_t kFormatCodes5 = 2;
constexpr int64_t kHeaderBytes = 256;

struct Codes5Header {
  uint32_t magic, format;
  int64_t n_out, k_red, n_chunks;
  uint32_t invalid_count, pad;
};

bool dims_in_range(int64_t n_out, int64_t k_red) {
  return n_out > 0 && k_red > 0 && n_out <= (int64_t(1) << 31) && k_red <= (int64_t(1) << 40) &&
         k_red <= (int64_t(1) << 48) / n_out;
}

int64_t records_end(int64_t n_out, int64_t k_red) { return kHeaderBytes + n_out * ((k_red + 31) / 32) * 20; }
int64_t blob_total(int64_t n_out, int64_t k_red) { return (records_end(n_out, k_red) + 255) / 256 * 256; }

__global__ void pack5_kernel(const int8_t* __restrict__ s, const int8_t* __restrict__ p, int64_t n_out,
                             int64_t k_red, int64_t n_chunks, uint32_t* __restrict__ rec, uint32_t* invalid) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = blockIdx.x * (int64_t)(blockDim.x >> 5) + (threadIdx.x >> 5); r < n_out * n_chunks;
       r += warps) {
    const int64_t n = r / n_chunks, k = (r - n * n_chunks) * 32 + lane;
    uint32_t c = 0;
    bool bad = false;
    if (k < k_red) {
      const int sv = s[n * k_red + k], pv = p[n * k_red + k];
      if (sv == 0 && pv >= -15 && pv <= 0)
        c = 0;
      else if ((sv == 1 || sv == -1) && pv >= -14 && pv <= 0)
        c = (sv == 1 ? 1u : 16u) + (uint32_t)(-pv);
      else
        bad = true;
    }
#pragma unroll
    for (int b = 0; b < 5; ++b) {
      const uint32_t w = __ballot_sync(0xffffffffu, (c >> b) & 1u);
      if (lane == b) rec[r * 5 + b] = w;
    }
    const int nbad = __popc(__ballot_sync(0xffffffffu, bad));
    if (lane == 0 && nbad) atomicAdd(invalid, (uint32_t)nbad);
  }
}

// Codes read back; code 31 (never written by the packer) becomes a zero weight and is counted.
__device__ uint32_t g_unpack5_invalid;

__global__ void unpack5_kernel(const uint32_t* __restrict__ rec, int64_t n_out, int64_t k_red, int64_t n_chunks,
                               int8_t* __restrict__ s, int8_t* __restrict__ p) {
  const int64_t total = n_out * k_red;
  uint32_t bad = 0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = e / k_red, k = e - n * k_red;
    const uint32_t* rr = rec + (n * n_chunks + (k >> 5)) * 5;
    const int j = (int)(k & 31);
    uint32_t c = 0;
#pragma unroll
    for (int b = 0; b < 5; ++b) c |= ((__ldg(rr + b) >> j) & 1u) << b;
    int sv = 0, pv = 0;
    if (c >= 1 && c <= 15) {
      sv = 1;
      pv = -(int)(c - 1);
    } else if (c >= 16 && c <= 30) {
      sv = -1;
      pv = -(int)(c - 16);
    } else if (c == 31) {
      ++bad;
    }
    s[e] = (int8_t)sv;
    p[e] = (int8_t)pv;
  }
  bad = __reduce_add_sync(0xffffffffu, bad);
  if ((threadIdx.x & 31) == 0 && bad) atomicAdd(&g_unpack5_invalid, bad);
}

int64_t grid_for(int64_t items, int threads) {
  const int64_t cap = (int64_t)(ds::sm_count() > 0 ? ds::sm_count() : 1) * 8;
  const int64_t b = (items + threads - 1) / threads;
  return b < 1 ? 1 : (b > cap ? cap : b);
}

std::mutex g_unpack_mutex;  // the invalid-code counter is one per device

}  // namespace

extern "C" {

size_t ds_packed5_weight_bytes(int64_t n_out, int64_t k_red) {
  if (!dims_in_range(n_out, k_red)) return 0;
  return (size_t)blob_total(n_out, k_red);
}

ds_status ds_pack_shift_weights5(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red, void* packed5,
                                 size_t packed5_bytes, void* stream) {
  ds::NvtxRange nvtx_range("ds_pack_shift_weights5");
  ds::clear_error();
  if (!s || !p || !packed5) return ds::fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n_out <= 0 || k_red <= 0) return ds::fail(DS_ERR_SHAPE, "n_out and k_red must be positive");
  const size_t need = ds_packed5_weight_bytes(n_out, k_red);
  if (need == 0) return ds::fail(DS_ERR_UNSUPPORTED, "code matrix too large");
  if (packed5_bytes < need)
    return ds::fail(DS_ERR_BUFFER_TOO_SMALL, "5-bit blob buffer has %zu bytes, needs %zu", packed5_bytes, need);
  if ((reinterpret_cast<uintptr_t>(packed5) & 255) != 0)
    return ds::fail(DS_ERR_ALIGNMENT, "5-bit blob buffer must be 256-byte aligned");
  if (ds::sm_count() <= 0) return ds::fail(DS_ERR_CUDA, "no CUDA device");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* blob = static_cast<uint8_t*>(packed5);
  const int64_t n_chunks = (k_red + 31) / 32;
  Codes5Header h{};
  h.magic = DS_WEIGHTS_MAGIC;
  h.format = kFormatCodes5;
  h.n_out = n_out;
  h.k_red = k_red;
  h.n_chunks = n_chunks;
  ds_status r = ds::cuda_check(cudaMemsetAsync(blob, 0, kHeaderBytes, st), "5-bit header reset");
  if (r == DS_OK) r = ds::cuda_check(cudaMemcpyAsync(blob, &h, sizeof(h), cudaMemcpyHostToDevice, st), "5-bit header");
  const int64_t end = records_end(n_out, k_red);
  if (r == DS_OK && (int64_t)need > end)
    r = ds::cuda_check(cudaMemsetAsync(blob + end, 0, need - end, st), "5-bit blob tail");
  if (r != DS_OK) return r;
  uint32_t* invalid = reinterpret_cast<uint32_t*>(blob + offsetof(Codes5Header, invalid_count));
  pack5_kernel<<<(unsigned)grid_for(n_out * n_chunks * 32, 256), 256, 0, st>>>(
      s, p, n_out, k_red, n_chunks, reinterpret_cast<uint32_t*>(blob + kHeaderBytes), invalid);
  r = ds::cuda_check(cudaGetLastError(), "5-bit pack launch");
  if (r != DS_OK) return r;
  uint32_t bad = 0;
  r = ds::cuda_check(cudaMemcpyAsync(&bad, invalid, sizeof(bad), cudaMemcpyDeviceToHost, st), "5-bit verdict");
  if (r == DS_OK) r = ds::cuda_check(cudaStreamSynchronize(st), "5-bit pack synchronise");
  if (r != DS_OK) return r;
  if (bad != 0)
    return ds::fail(DS_ERR_CODE_RANGE, "%u codes outside the 5-bit states (s in {-1,0,1}; p in [-14,0] when s != 0)",
                    bad);
  return DS_OK;
}

ds_status ds_unpack_shift_weights5(const void* packed5, size_t packed5_bytes, int64_t n_out, int64_t k_red,
                                   int8_t* s, int8_t* p, void* stream) {
  ds::NvtxRange nvtx_range("ds_unpack_shift_weights5");
  ds::clear_error();
  if (!packed5 || !s || !p) return ds::fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n_out <= 0 || k_red <= 0) return ds::fail(DS_ERR_SHAPE, "n_out and k_red must be positive");
  const size_t need = ds_packed5_weight_bytes(n_out, k_red);
  if (need == 0) return ds::fail(DS_ERR_UNSUPPORTED, "code matrix too large");
  if (packed5_bytes < need)
    return ds::fail(DS_ERR_BUFFER_TOO_SMALL, "5-bit blob has %zu bytes, needs %zu", packed5_bytes, need);
  if ((reinterpret_cast<uintptr_t>(packed5) & 255) != 0)
    return ds::fail(DS_ERR_ALIGNMENT, "5-bit blob must be 256-byte aligned");
  if (ds::sm_count() <= 0) return ds::fail(DS_ERR_CUDA, "no CUDA device");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Codes5Header h{};
  ds_status r = ds::cuda_check(cudaMemcpyAsync(&h, packed5, sizeof(h), cudaMemcpyDeviceToHost, st), "5-bit header");
  if (r == DS_OK) r = ds::cuda_check(cudaStreamSynchronize(st), "5-bit header read");
  if (r != DS_OK) return r;
  const int64_t n_chunks = (k_red + 31) / 32;
  if (h.magic != DS_WEIGHTS_MAGIC || h.format != kFormatCodes5)
    return ds::fail(DS_ERR_INVALID_ARG, "not a 5-bit blob written by ds_pack_shift_weights5");
  if (h.n_out != n_out || h.k_red != k_red || h.n_chunks != n_chunks)
    return ds::fail(DS_ERR_SHAPE, "5-bit blob holds %lld x %lld codes, call asks for %lld x %lld",
                    (long long)h.n_out, (long long)h.k_red, (long long)n_out, (long long)k_red);
  std::lock_guard<std::mutex> lock(g_unpack_mutex);
  const uint32_t zero = 0;
  r = ds::cuda_check(cudaMemcpyToSymbolAsync(g_unpack5_invalid, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st),
                     "5-bit counter reset");
  if (r != DS_OK) return r;
  unpack5_kernel<<<(unsigned)grid_for(n_out * k_red, 256), 256, 0, st>>>(
      reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(packed5) + kHeaderBytes), n_out, k_red, n_chunks,
      s, p);
  r = ds::cuda_check(cudaGetLastError(), "5-bit unpack launch");
  if (r != DS_OK) return r;
  uint32_t bad = 0;
  r = ds::cuda_check(cudaMemcpyFromSymbolAsync(&bad, g_unpack5_invalid, sizeof(bad), 0, cudaMemcpyDeviceToHost, st),
                     "5-bit verdict");
  if (r == DS_OK) r = ds::cuda_check(cudaStreamSynchronize(st), "5-bit unpack synchronise");
  if (r != DS_OK) return r;
  if (bad != 0) return ds::fail(DS_ERR_CODE_RANGE, "%u codes of the 5-bit blob are 31 (never written)", bad);
  return DS_OK;
}

}  // extern "C"
