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
      // the lane's 4 codes decoded a byte at a time with SIMD-in-word operations
      const uint32_t inm = in ? 0xffffffffu : 0u;
      const uint32_t bad = (__vcmpgtu4(__vadd4(sw, 0x01010101u), 0x02020202u) |   // s outside {-1, 0, 1}
                            __vcmpgtu4(__vadd4(pw, 0x0f0f0f0fu), 0x0f0f0f0fu)) &  // p outside [-15, 0]
                           inm;
      const uint32_t okm = inm & ~bad;
      invalid += (uint32_t)__popc(bad & 0x01010101u);
      const uint32_t nzm = __vcmpne4(sw, 0u) & okm;              // s != 0
      const uint32_t ngm = __vcmpeq4(sw, 0xffffffffu) & okm;     // s == -1
      // byte masks (0x00 / 0xff) to 4 bits: (m & 0x01010101) * 0x10204080 >> 28
      const uint32_t zb = ((nzm & 0x01010101u) * 0x10204080u) >> 28;
      const uint32_t nb = ((ngm & 0x01010101u) * 0x10204080u) >> 28;
      // shift nibbles k = -p: byte i of q holds k_i; packed as bits 4i .. 4i + 3
      const uint32_t q = __vsub4(0u, pw) & okm;
      const uint32_t nib = __byte_perm(q | (q >> 4), 0u, 0x4420u);  // bytes 0 and 2, then zeros
      // A: sum of 2^(15 - k) over the nonzero codes, as 2^8 * sum 2^(7 - k) (k < 8) + sum 2^(15 - k) (k >= 8);
      // each byte's power of two 2^(7 - (k & 7)) from a byte table selected by k & 7
      const uint32_t pw2 = __byte_perm(0x10204080u, 0x01020408u, nib & 0x7777u) & nzm;
      const uint32_t hi = __vcmpltu4(q, 0x08080808u);
      const uint32_t a_sum = (__vsadu4(pw2 & hi, 0u) << 8) + __vsadu4(pw2 & ~hi, 0u);
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

// Decode of 4 codes held as the bytes of one word of s and one of p (SIMD
// in word): the out-of-range count, the non-zero and negative bits (bit i for
// byte i), the 4 shift nibbles (bits 4i .. 4i + 3) and the codes' share of A.
struct Quad {
  uint32_t bad, zb, nb, nib, a;
};
__device__ __forceinline__ Quad decode_quad(uint32_t sw, uint32_t pw) {
  Quad r;
  const uint32_t bad = __vcmpgtu4(__vadd4(sw, 0x01010101u), 0x02020202u) |  // s outside {-1, 0, 1}
                       __vcmpgtu4(__vadd4(pw, 0x0f0f0f0fu), 0x0f0f0f0fu);   // p outside [-15, 0]
  const uint32_t okm = ~bad;
  const uint32_t nzm = __vcmpne4(sw, 0u) & okm;
  const uint32_t ngm = __vcmpeq4(sw, 0xffffffffu) & okm;
  r.bad = (uint32_t)__popc(bad & 0x01010101u);
  r.zb = ((nzm & 0x01010101u) * 0x10204080u) >> 28;  // byte masks to 4 bits
  r.nb = ((ngm & 0x01010101u) * 0x10204080u) >> 28;
  const uint32_t q = __vsub4(0u, pw) & okm;            // k = -p per byte
  r.nib = __byte_perm(q | (q >> 4), 0u, 0x4420u);
  // 2^(15 - k) = 2^8 * 2^(7 - k) for k < 8, else 2^(7 - (k - 8)): a byte table selected by k & 7
  const uint32_t pw2 = __byte_perm(0x10204080u, 0x01020408u, r.nib & 0x7777u) & nzm;
  const uint32_t hi = __vcmpltu4(q, 0x08080808u);
  r.a = (__vsadu4(pw2 & hi, 0u) << 8) + __vsadu4(pw2 & ~hi, 0u);
  return r;
}

// Packing with 16 codes per lane (k_red a multiple of 16, 16-byte aligned
// rows): one 16-byte load of s and one of p per lane; a 32-code chunk is a
// lane pair, whose even lane writes the chunk's first two shift words and the
// bit planes, the odd lane the last two shift words.  A warp covers 512
// codes of one column per step.
__global__ void pack_kernel_vec16(const int8_t* __restrict__ s, const int8_t* __restrict__ p, int64_t n_out,
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
  const int64_t steps = (k_red + 511) / 512;
  const int64_t per = (steps + parts - 1) / parts;
  const int64_t units = n_out * parts;
  uint2* nibw = reinterpret_cast<uint2*>(blob + L.nib);
  uint2* bits = reinterpret_cast<uint2*>(blob + L.bits);
  for (int64_t u = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; u < units;
       u += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t n = u % n_out;
    const int64_t b0 = (u / n_out) * per;
    const int64_t b1 = b0 + per < steps ? b0 + per : steps;
    const uint4* srow = reinterpret_cast<const uint4*>(s + n * k_red);
    const uint4* prow = reinterpret_cast<const uint4*>(p + n * k_red);
    uint32_t nnz = 0, invalid = 0;
    unsigned long long a_col = 0;
    for (int64_t b = b0; b < b1; b += 2) {  // two steps' loads in flight
      uint4 sv[2], pv[2];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const bool in = b + q < b1 && (b + q) * 512 + 16 * lane < k_red;
        sv[q] = in ? __ldg(srow + (b + q) * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
        pv[q] = in ? __ldg(prow + (b + q) * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        if (b + q >= b1) break;
        const Quad d0 = decode_quad(sv[q].x, pv[q].x), d1 = decode_quad(sv[q].y, pv[q].y);
        const Quad d2 = decode_quad(sv[q].z, pv[q].z), d3 = decode_quad(sv[q].w, pv[q].w);
        invalid += d0.bad + d1.bad + d2.bad + d3.bad;
        const uint32_t zb = d0.zb | (d1.zb << 4) | (d2.zb << 8) | (d3.zb << 12);
        const uint32_t nb = d0.nb | (d1.nb << 4) | (d2.nb << 8) | (d3.nb << 12);
        nnz += (uint32_t)__popc(zb);
        const uint32_t a_sum = d0.a + d1.a + d2.a + d3.a;  // at most 16 * 2^15
        // planes of the lane pair's chunk: the even lane's 16 codes in bits 0..15, the odd lane's in 16..31
        const int sh = 16 * (lane & 1);
        uint32_t np = nb << sh, zp = zb << sh;
        np |= __shfl_xor_sync(full, np, 1);
        zp |= __shfl_xor_sync(full, zp, 1);
        const int64_t g = (b + q) * 16 + (lane >> 1);  // this lane's chunk
        if (g < L.n_chunks) {
          // shift words 2 (lane & 1), 2 (lane & 1) + 1 of the chunk
          nibw[((g * n_out + n) * 4 + 2 * (lane & 1)) >> 1] =
              make_uint2(d0.nib | (d1.nib << 16), d2.nib | (d3.nib << 16));
          if ((lane & 1) == 0) bits[g * n_out + n] = make_uint2(np, zp);
        }
        a_col += __reduce_add_sync(full, a_sum);  // a warp step adds at most 2^24
      }
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
  const bool vec16 = vec4 && (k_red % 16) == 0 && (reinterpret_cast<uintptr_t>(s) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(p) & 15) == 0;
  // zero the header counters, the column constants (added atomically) and the tail padding; the vectorised
  // kernels write every shift word and bit plane, the general one gets the whole blob zeroed
  const BlobLayout L = blob_layout(n_out, k_red);
  cudaError_t e;
  if (vec4) {
    e = cudaMemsetAsync(blob, 0, (size_t)L.nib, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(blob + L.col_a, 0, (size_t)(L.total - L.col_a), st);
  } else {
    e = cudaMemsetAsync(blob, 0, (size_t)L.total, st);
  }
  if (e != cudaSuccess) return e;
  if (vec4) {  // 128- or 512-index steps: split a column's steps into parts the same way
    const int64_t steps = vec16 ? (k_red + 511) / 512 : (k_red + 127) / 128;
    if (parts > steps) parts = steps;
  }
  const int64_t units = n_out * parts;
  int64_t blocks = (units + threads / 32 - 1) / (threads / 32);
  if (blocks > (int64_t)sms * 32) blocks = (int64_t)sms * 32;  // grid-stride beyond
  if (vec16) {
    pack_kernel_vec16<<<(unsigned)blocks, threads, 0, st>>>(s, p, n_out, k_red, blob, parts);
  } else if (vec4) {
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
