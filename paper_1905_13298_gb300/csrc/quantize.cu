// Float -> shift code (DeepShift-Q, Eq. 4-6) and float -> Q16.16 (Sec. 4).
//
// Weights: s = sign(W), p = clip(round(log2|W|), p_min, 0).  For a normal
// float32 W with biased exponent E and 24-bit significand m (|W| =
// m 2^(E - 150)), log2|W| = (E - 127) + log2(m / 2^23) with m / 2^23 in
// [1, 2); the fraction rounds up exactly when (m / 2^23)^2 >= 2, i.e.
// m^2 >= 2^47 (a 64-bit integer comparison; the bound sqrt(2) is
// irrational, so there are no ties).  Zero and NaN give s = 0, p = p_min;
// +-inf give s = +-1, p = 0; subnormals (|W| < 2^-126) give p = p_min.
//
// Activations: q = rint(x * 2^16) (ties to even; the scaling is exact),
// saturated to the int32 range, NaN -> 0.
//
// Both are streaming kernels bound by HBM with four independent 16-byte loads
// in flight per thread and 16-byte stores, a grid of 8 CTAs per SM striding
// over the array.
#include "ds_common.cuh"

namespace ds {
namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;
constexpr int kUnroll = 4;  // independent 16-byte loads in flight per thread

struct Code {
  int8_t s, p;
};

__device__ __forceinline__ Code code_of(uint32_t bits, int p_min) {
  const uint32_t ex = (bits >> 23) & 0xFFu;
  const uint32_t man = bits & 0x7FFFFFu;
  const int8_t sg = (bits >> 31) ? (int8_t)-1 : (int8_t)1;
  if (ex == 0xFFu) return man ? Code{0, (int8_t)p_min} : Code{sg, 0};      // NaN, +-inf
  if (ex == 0u) return man ? Code{sg, (int8_t)p_min} : Code{0, (int8_t)p_min};  // subnormal, zero
  const uint64_t m = (1ull << 23) | man;
  const int r = (int)ex - 127 + ((m * m >= (1ull << 47)) ? 1 : 0);  // round(log2|W|), Eq. 5
  return Code{sg, (int8_t)(r < p_min ? p_min : (r > 0 ? 0 : r))};
}

__device__ __forceinline__ int32_t q16_of(float x) {
  if (x != x) return 0;
  const float y = rintf(x * 65536.0f);
  if (y >= 2147483648.0f) return INT32_MAX;
  if (y < -2147483648.0f) return INT32_MIN;
  return (int32_t)y;
}

__device__ __forceinline__ uint32_t pack4(int8_t a, int8_t b, int8_t c, int8_t d) {
  return (uint32_t)(uint8_t)a | ((uint32_t)(uint8_t)b << 8) | ((uint32_t)(uint8_t)c << 16) |
         ((uint32_t)(uint8_t)d << 24);
}

// VEC: a thread converts 16 consecutive weights per step (four 16-byte
// loads, all in flight before the first use) and writes each code stream
// with one 16-byte store.
template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_weights_kernel(const float* __restrict__ w, int64_t n,
                                                                    int p_min, int8_t* __restrict__ s,
                                                                    int8_t* __restrict__ p) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t done = 0;
  if constexpr (VEC) {
    const int64_t n16 = n / 16;
    for (int64_t i = tid; i < n16; i += stride) {
      uint4 b[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) b[u] = __ldg(reinterpret_cast<const uint4*>(w) + 4 * i + u);
      uint32_t ws[4], wp[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const Code c0 = code_of(b[u].x, p_min), c1 = code_of(b[u].y, p_min), c2 = code_of(b[u].z, p_min),
                   c3 = code_of(b[u].w, p_min);
        ws[u] = pack4(c0.s, c1.s, c2.s, c3.s);
        wp[u] = pack4(c0.p, c1.p, c2.p, c3.p);
      }
      reinterpret_cast<uint4*>(s)[i] = make_uint4(ws[0], ws[1], ws[2], ws[3]);
      reinterpret_cast<uint4*>(p)[i] = make_uint4(wp[0], wp[1], wp[2], wp[3]);
    }
    done = n16 * 16;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    const Code c = code_of(__float_as_uint(__ldg(w + i)), p_min);
    s[i] = c.s;
    p[i] = c.p;
  }
}

template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_q16_kernel(const float* __restrict__ x, int64_t n,
                                                                int32_t* __restrict__ q) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t done = 0;
  if constexpr (VEC) {
    const int64_t n4 = n / 4;
    for (int64_t i = tid; i < n4; i += stride * kUnroll) {
      float4 v[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t j = i + u * stride;
        if (j < n4) v[u] = __ldg(reinterpret_cast<const float4*>(x) + j);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t j = i + u * stride;
        if (j < n4) reinterpret_cast<int4*>(q)[j] = make_int4(q16_of(v[u].x), q16_of(v[u].y), q16_of(v[u].z),
                                                              q16_of(v[u].w));
      }
    }
    done = n4 * 4;
  }
  for (int64_t i = done + tid; i < n; i += stride) q[i] = q16_of(__ldg(x + i));
}

unsigned grid_for(int64_t n) {
  const int64_t want = (n / 4 + (int64_t)kThreads * kUnroll - 1) / ((int64_t)kThreads * kUnroll);
  const int64_t cap = (int64_t)(sm_count() > 0 ? sm_count() : 1) * kBlocksPerSm;
  return (unsigned)(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

cudaError_t launch_quantize_weights(const float* w, int64_t n, int p_min, int8_t* s, int8_t* p, cudaStream_t st) {
  const bool vec = ((reinterpret_cast<uintptr_t>(w) & 15) == 0) && ((reinterpret_cast<uintptr_t>(s) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(p) & 15) == 0);
  if (vec) {
    quantize_weights_kernel<true><<<grid_for(n / 4), kThreads, 0, st>>>(w, n, p_min, s, p);
  } else {
    quantize_weights_kernel<false><<<grid_for(n), kThreads, 0, st>>>(w, n, p_min, s, p);
  }
  return cudaGetLastError();
}

cudaError_t launch_quantize_q16(const float* x, int64_t n, int32_t* q, cudaStream_t st) {
  const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && ((reinterpret_cast<uintptr_t>(q) & 15) == 0);
  if (vec) {
    quantize_q16_kernel<true><<<grid_for(n), kThreads, 0, st>>>(x, n, q);
  } else {
    quantize_q16_kernel<false><<<grid_for(n), kThreads, 0, st>>>(x, n, q);
  }
  return cudaGetLastError();
}

}  // namespace ds
