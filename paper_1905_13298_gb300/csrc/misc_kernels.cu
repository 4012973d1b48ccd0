// Weight packing and the max|x| pre-pass.
//
// Packing follows Eq. 3 of DeepShift (the weight matrix is replaced by the
// shift matrix P and the sign matrix S) with the Sec. 4 range p in [-15, 0];
// the blob layout is the library's own (deepshift.h, DS_FORMAT_PLANES6).
#include "ds_common.cuh"

namespace ds {

struct BwdMap {
  int K, C, R, S, sh, sw, a, b, Th, Tw;  // K == 0: forward layout
};

// One warp per (column n, range of 32-index chunks).  Lane j holds code j of
// a chunk: with the forward layout the warp's two loads are 32 consecutive
// bytes of row n (coalesced).  The chunk's records come from warp votes (sign
// and non-zero planes) and an OR over each group of 8 lanes (the four shift
// words); lane 0 writes them.  Records of consecutive columns are adjacent,
// and consecutive warps take consecutive columns, so the writes of a block
// merge.  Per-column constants A[n], nnz[n] and the invalid count are added
// atomically (the blob starts zeroed); pack_maxima_kernel then folds the
// columns into the header maxima.
__global__ void pack_kernel(const int8_t* __restrict__ s, const int8_t* __restrict__ p, int64_t n_out,
                            int64_t k_red, uint8_t* __restrict__ blob, const BwdMap m, int64_t parts) {
  const BlobLayout L = blob_layout(n_out, k_red);
  BlobHeader* hdr = reinterpret_cast<BlobHeader*>(blob);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    hdr->magic = DS_WEIGHTS_MAGIC;
    hdr->format = DS_FORMAT_PLANES6;
    hdr->n_out = n_out;
    hdr->k_red = k_red;
    hdr->n_chunks = L.n_chunks;
  }
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int64_t per = (L.n_chunks + parts - 1) / parts;  // chunks per warp
  const int64_t units = n_out * parts;
  const int64_t tt = (int64_t)m.Th * m.Tw;
  uint4* nib = reinterpret_cast<uint4*>(blob + L.nib);
  uint2* bits = reinterpret_cast<uint2*>(blob + L.bits);
  for (int64_t u = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; u < units;
       u += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t n = u % n_out;
    const int64_t g0 = (u / n_out) * per;
    const int64_t g1 = g0 + per < L.n_chunks ? g0 + per : L.n_chunks;
    // forward: column n's codes are row n.  Input-gradient phase (m.K > 0):
    // column n is input channel n, index k = (k_out, t, u) reads the code of
    // tap (m.a + m.sh (Th-1-t), m.b + m.sw (Tw-1-u)) of (k_out, n)
    auto offset = [&](int64_t k) -> int64_t {
      if (m.K == 0) return n * k_red + k;
      const int64_t ko = k / tt, rem = k - ko * tt;
      const int64_t t = rem / m.Tw, v = rem - t * m.Tw;
      const int64_t r = m.a + (int64_t)m.sh * (m.Th - 1 - t), q = m.b + (int64_t)m.sw * (m.Tw - 1 - v);
      return ((ko * m.C + n) * m.R + r) * m.S + q;
    };
    unsigned long long a_sum = 0;
    uint32_t nnz = 0, invalid = 0;
#pragma unroll 4
    for (int64_t g = g0; g < g1; ++g) {
      const int64_t k = g * kChunk + lane;
      int sv = 0, pv = 0;
      const bool in = k < k_red;
      if (in) {
        const int64_t o = offset(k);
        sv = s[o];
        pv = p[o];
      }
      const bool bad = in && (sv < -1 || sv > 1 || pv < -15 || pv > 0);
      const bool ok = in && !bad;
      const uint32_t neg = __ballot_sync(full, ok && sv == -1);
      const uint32_t nz = __ballot_sync(full, ok && sv != 0);
      const uint32_t badm = __ballot_sync(full, bad);
      uint32_t w = ok ? (uint32_t)(-pv) << (4 * (lane & 7)) : 0u;
      w |= __shfl_xor_sync(full, w, 1);
      w |= __shfl_xor_sync(full, w, 2);
      w |= __shfl_xor_sync(full, w, 4);
      const uint32_t w1 = __shfl_sync(full, w, 8), w2 = __shfl_sync(full, w, 16), w3 = __shfl_sync(full, w, 24);
      const uint32_t a = __reduce_add_sync(full, (ok && sv != 0) ? (1u << (15 + pv)) : 0u);  // <= 2^20
      if (lane == 0) {
        nib[g * n_out + n] = make_uint4(w, w1, w2, w3);
        bits[g * n_out + n] = make_uint2(neg, nz);
      }
      a_sum += a;
      nnz += (uint32_t)__popc(nz);
      invalid += (uint32_t)__popc(badm);
    }
    if (lane == 0) {
      atomicAdd(reinterpret_cast<unsigned long long*>(blob + L.col_a) + n, a_sum);
      atomicAdd(reinterpret_cast<uint32_t*>(blob + L.nnz) + n, nnz);
      if (invalid) atomicAdd(&hdr->invalid_count, invalid);
    }
  }
}

// Forward layout with 4-byte aligned rows (k_red % 4 == 0, s and p 4-byte
// aligned): the same records, 128 reduction indices (4 chunks) per warp step.
// Lane j loads codes 4j .. 4j + 3 of the step with one 32-bit load of s and
// one of p, so lanes 8q .. 8q + 7 hold chunk q.  Each lane forms its 4 codes'
// plane bits and nibbles; ORs over each group of 8 lanes (planes) and over
// lane pairs (the shift word of 8 codes) assemble the records; lanes 8q + 2w
// write shift word w of chunk q and lane 8q writes its bit planes.
__global__ void pack_kernel_vec4(const int8_t* __restrict__ s, const int8_t* __restrict__ p, int64_t n_out,
                                 int64_t k_red, uint8_t* __restrict__ blob, int64_t parts) {
  const BlobLayout L = blob_layout(n_out, k_red);
  BlobHeader* hdr = reinterpret_cast<BlobHeader*>(blob);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    hdr->magic = DS_WEIGHTS_MAGIC;
    hdr->format = DS_FORMAT_PLANES6;
    hdr->n_out = n_out;
    hdr->k_red = k_red;
    hdr->n_chunks = L.n_chunks;
  }
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int jj = lane & 7;  // lane within its chunk's group
  const int64_t steps = (k_red + 127) / 128;
  const int64_t per = (steps + parts - 1) / parts;
  const int64_t units = n_out * parts;
  uint32_t* nibw = reinterpret_cast<uint32_t*>(blob + L.nib);
  uint2* bits = reinterpret_cast<uint2*>(blob + L.bits);
  for (int64_t u = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; u < units;
       u += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t n = u % n_out;
    const int64_t b0 = (u / n_out) * per;
    const int64_t b1 = b0 + per < steps ? b0 + per : steps;
    const uint32_t* srow = reinterpret_cast<const uint32_t*>(s + n * k_red);
    const uint32_t* prow = reinterpret_cast<const uint32_t*>(p + n * k_red);
    uint32_t nnz = 0, invalid = 0;  // per lane
    unsigned long long a_col = 0;
    // one warp step: 128 indices of the column from the lane's words sw, pw
    auto step = [&](int64_t b, uint32_t sw, uint32_t pw) {
      const int64_t k0 = b * 128 + 4 * lane;
      const bool in = k0 < k_red;  // k_red % 4 == 0: all 4 codes or none
      uint32_t nb = 0u, zb = 0u, nib = 0u, a_sum = 0u;  // a lane adds at most 2^15 per code
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int sv = (int)(int8_t)(sw >> (8 * i));
        const int pv = (int)(int8_t)(pw >> (8 * i));
        const bool bad = in && ((unsigned)(sv + 1) > 2u || (unsigned)(pv + 15) > 15u);
        const bool ok = in && !bad;
        invalid += bad ? 1u : 0u;
        if (ok) {
          nib |= (uint32_t)(-pv) << (4 * i);
          if (sv != 0) {
            zb |= 1u << i;
            a_sum += 1u << (15 + pv);
          }
          if (sv == -1) nb |= 1u << i;
        }
      }
      nnz += (uint32_t)__popc(zb);
      // planes of chunk q: lane 8q + jj holds bits 4 jj .. 4 jj + 3
      uint32_t np = nb << (4 * jj), zp = zb << (4 * jj);
      np |= __shfl_xor_sync(full, np, 1);
      zp |= __shfl_xor_sync(full, zp, 1);
      np |= __shfl_xor_sync(full, np, 2);
      zp |= __shfl_xor_sync(full, zp, 2);
      np |= __shfl_xor_sync(full, np, 4);
      zp |= __shfl_xor_sync(full, zp, 4);
      // shift word w (codes 8w .. 8w + 7) of chunk q: lanes 8q + 2w, 8q + 2w + 1
      uint32_t w = nib << (16 * (jj & 1));
      w |= __shfl_xor_sync(full, w, 1);
      const int64_t g = b * 4 + (lane >> 3);  // this lane's chunk
      if (g < L.n_chunks) {
        if ((jj & 1) == 0) nibw[(g * n_out + n) * 4 + (jj >> 1)] = w;
        if (jj == 0) bits[g * n_out + n] = make_uint2(np, zp);
      }
      a_col += __reduce_add_sync(full, a_sum);  // a warp step adds at most 2^22
    };
    // four steps per iteration, their loads issued before any is decoded
    for (int64_t b = b0; b < b1; b += 4) {
      uint32_t sw[4], pw[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const bool in = b + q < b1 && (b + q) * 128 + 4 * lane < k_red;
        sw[q] = in ? __ldg(srow + (((b + q) * 128) >> 2) + lane) : 0u;
        pw[q] = in ? __ldg(prow + (((b + q) * 128) >> 2) + lane) : 0u;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (b + q < b1) step(b + q, sw[q], pw[q]);
    }
    nnz = __reduce_add_sync(full, nnz);
    invalid = __reduce_add_sync(full, invalid);
    if (lane == 0) {
      atomicAdd(reinterpret_cast<unsigned long long*>(blob + L.col_a) + n, a_col);
      atomicAdd(reinterpret_cast<uint32_t*>(blob + L.nnz) + n, nnz);
      if (invalid) atomicAdd(&hdr->invalid_count, invalid);
    }
  }
}

// Header maxima over the columns' A[n] and nnz[n].
__global__ void pack_maxima_kernel(uint8_t* __restrict__ blob, int64_t n_out, int64_t k_red) {
  const BlobLayout L = blob_layout(n_out, k_red);
  BlobHeader* hdr = reinterpret_cast<BlobHeader*>(blob);
  const unsigned long long* A = reinterpret_cast<const unsigned long long*>(blob + L.col_a);
  const uint32_t* nz = reinterpret_cast<const uint32_t*>(blob + L.nnz);
  unsigned long long am = 0;
  uint32_t nm = 0;
  for (int64_t n = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; n < n_out; n += (int64_t)gridDim.x * blockDim.x) {
    am = A[n] > am ? A[n] : am;
    nm = nz[n] > nm ? nz[n] : nm;
  }
  nm = __reduce_max_sync(0xffffffffu, nm);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const unsigned long long v = __shfl_xor_sync(0xffffffffu, am, o);
    am = v > am ? v : am;
  }
  if ((threadIdx.x & 31) == 0) {
    if (nm) atomicMax(&hdr->nnz_max, nm);
    if (am) atomicMax(&hdr->a_max, am);
  }
}

cudaError_t launch_pack(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red,
                        uint8_t* blob, cudaStream_t st, const int* bwd) {
  // zero the whole blob: header counters, column constants (added atomically), tail padding
  cudaError_t e = cudaMemsetAsync(blob, 0, (size_t)blob_layout(n_out, k_red).total, st);
  if (e != cudaSuccess) return e;
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorNoDevice;
  BwdMap m{0, 0, 1, 1, 1, 1, 0, 0, 1, 1};
  if (bwd != nullptr) m = BwdMap{bwd[0], bwd[1], bwd[2], bwd[3], bwd[4], bwd[5], bwd[6], bwd[7], bwd[8], bwd[9]};
  // enough warps for 64 per SM: split each column's chunks into parts when there are few columns
  const int threads = 256;
  const int64_t n_chunks = blob_layout(n_out, k_red).n_chunks;
  const int64_t want = (int64_t)sms * 64;
  int64_t parts = (want + n_out - 1) / n_out;
  if (parts > n_chunks) parts = n_chunks;
  if (parts < 1) parts = 1;
  const bool vec4 = bwd == nullptr && (k_red % 4) == 0 && (reinterpret_cast<uintptr_t>(s) & 3) == 0 &&
                    (reinterpret_cast<uintptr_t>(p) & 3) == 0;
  if (vec4) {  // 128-index steps: split a column's steps into parts the same way
    const int64_t steps = (k_red + 127) / 128;
    if (parts > steps) parts = steps;
  }
  const int64_t units = n_out * parts;
  int64_t blocks = (units + threads / 32 - 1) / (threads / 32);
  if (blocks > (int64_t)sms * 32) blocks = (int64_t)sms * 32;  // grid-stride beyond
  if (vec4) {
    pack_kernel_vec4<<<(unsigned)blocks, threads, 0, st>>>(s, p, n_out, k_red, blob, parts);
  } else {
    pack_kernel<<<(unsigned)blocks, threads, 0, st>>>(s, p, n_out, k_red, blob, m, parts);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int64_t mb = (n_out + threads - 1) / threads;
  if (mb > (int64_t)sms * 8) mb = (int64_t)sms * 8;
  pack_maxima_kernel<<<(unsigned)mb, threads, 0, st>>>(blob, n_out, k_red);
  return cudaGetLastError();
}

// Expanded execution layout: out[cb][k][c] = -p (c < 32) or s (c >= 32) of
// column 32*cb + (c & 31) at reduction index k; zero beyond n_out.
__global__ void expand_kernel(const uint8_t* __restrict__ blob, int64_t n_out, int64_t k_red,
                              int32_t* __restrict__ out) {
  const BlobLayout L = blob_layout(n_out, k_red);
  const int64_t total = ((n_out + 31) / 32) * k_red * 32;  // (cb, k, c32) triples
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int c32 = (int)(e & 31);
    const int64_t kc = e >> 5;  // cb * k_red + k
    const int64_t cb = kc / k_red;
    const int64_t k = kc - cb * k_red;
    const int64_t col = cb * 32 + c32;
    int32_t sh = 0, sg = 0;
    if (col < n_out) {
      const int64_t rec = (k >> 5) * n_out + col;
      const uint32_t nib = reinterpret_cast<const uint32_t*>(blob + L.nib + rec * 16)[(k >> 3) & 3];
      const uint2 b = reinterpret_cast<const uint2*>(blob + L.bits + rec * 8)[0];
      const int j = (int)(k & 31);
      sh = (int32_t)((nib >> (4 * (k & 7))) & 15u);
      sg = (int32_t)((b.y >> j) & 1u) - 2 * (int32_t)((b.x >> j) & 1u);
    }
    int32_t* row = out + kc * 64;
    row[c32] = sh;
    row[32 + c32] = sg;
  }
}

cudaError_t launch_expand(const uint8_t* blob, int64_t n_out, int64_t k_red, int32_t* out, cudaStream_t st) {
  const int threads = 256;
  const int64_t total = ((n_out + 31) / 32) * k_red * 32;
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > 65535 * 8) blocks = 65535 * 8;
  expand_kernel<<<(unsigned)blocks, threads, 0, st>>>(blob, n_out, k_red, out);
  return cudaGetLastError();
}

// max |x| (as u32, |INT32_MIN| = 2^31).  Grid-stride over 16-byte vectors,
// warp reduction, one atomicMax per warp.  The target is zeroed first.

__global__ void absmax_kernel(const int32_t* __restrict__ x, int64_t n, uint32_t* out) {
  uint32_t m = 0;
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15) == 0);
  if (vec) {
    const int64_t nv = n >> 2;
    const int4* xv = reinterpret_cast<const int4*>(x);
    int64_t i = tid;
    // eight independent 16-byte loads in flight per thread
    for (; i + 7 * stride < nv; i += 8 * stride) {
      int4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(xv + i + u * stride);
#pragma unroll
      for (int u = 0; u < 8; ++u) m = max(m, max(max(uabs(v[u].x), uabs(v[u].y)), max(uabs(v[u].z), uabs(v[u].w))));
    }
    for (; i < nv; i += stride) {
      const int4 a = __ldg(xv + i);
      m = max(m, max(max(uabs(a.x), uabs(a.y)), max(uabs(a.z), uabs(a.w))));
    }
    for (int64_t j = (nv << 2) + tid; j < n; j += stride) m = max(m, uabs(x[j]));
  } else {
    for (int64_t i = tid; i < n; i += stride) m = max(m, uabs(x[i]));
  }
  // block reduction, then one atomic per block
  __shared__ uint32_t wmax[32];
  m = __reduce_max_sync(0xffffffffu, m);
  if ((threadIdx.x & 31) == 0) wmax[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x < 32) {
    uint32_t v = threadIdx.x < (blockDim.x >> 5) ? wmax[threadIdx.x] : 0u;
    v = __reduce_max_sync(0xffffffffu, v);
    if (threadIdx.x == 0 && v) atomicMax(out, v);
  }
}

int sm_count() {
  // read once per process (thread-safe function-local static); the library
  // serves one device per process
  static const int sms = [] {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
                                                  cudaSuccess) {
      (void)cudaGetLastError();
      return 0;
    }
    return n;
  }();
  return sms;
}

cudaError_t launch_absmax(const int32_t* x, int64_t n, uint32_t* out, cudaStream_t st) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorNoDevice;
  cudaError_t e = cudaMemsetAsync(out, 0, sizeof(uint32_t), st);
  if (e != cudaSuccess) return e;
  const int threads = 256;
  int64_t want = (n / 16 + threads - 1) / threads;
  int64_t blocks = want < (int64_t)sms * 4 ? want : (int64_t)sms * 4;
  if (blocks < 1) blocks = 1;
  absmax_kernel<<<(unsigned)blocks, threads, 0, st>>>(x, n, out);
  return cudaGetLastError();
}

}  // namespace ds
