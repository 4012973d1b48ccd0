// Integer pooling for the chained forward of ResNet / VGG shaped networks
// (the pools around the shift layers of Eq. 3; the paper does not define
// them on fixed point).  Max-pool ignores padded taps; average pool is
// floor(sum / (R*S)) over a window without padding (floor division, also for
// negative sums).
#include "ds_common.cuh"

namespace ds {

// Output e = (plane, oh, ow) of a pool: below 2^31 outputs the coordinates
// come from two multiply-shift divisions, else from 64-bit ones.
struct PoolIndex {
  FastDiv d_ow, d_oh;
  bool fast;
};
__device__ __forceinline__ void pool_coords(int64_t e, int OH, int OW, const PoolIndex& ix, int64_t& pl, int& oh,
                                            int& ow) {
  if (ix.fast) {
    const int t = fdiv((int)e, ix.d_ow);
    ow = (int)e - t * OW;
    const int p = fdiv(t, ix.d_oh);
    oh = t - p * OH;
    pl = p;
  } else {
    ow = (int)(e % OW);
    const int64_t t = e / OW;
    oh = (int)(t % OH);
    pl = t / OH;
  }
}

__global__ void maxpool_kernel(const int32_t* __restrict__ x, int32_t* __restrict__ y, int64_t planes,
                               int H, int W, int OH, int OW, int R, int S, int stride, int pad, PoolIndex ix) {
  const int64_t total = planes * OH * OW;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    int64_t pl;
    int oh, ow;
    pool_coords(e, OH, OW, ix, pl, oh, ow);
    const int32_t* xp = x + pl * H * W;
    int32_t m = INT32_MIN;
    for (int r = 0; r < R; ++r) {
      const int ih = oh * stride - pad + r;
      if ((unsigned)ih >= (unsigned)H) continue;
      for (int s = 0; s < S; ++s) {
        const int iw = ow * stride - pad + s;
        if ((unsigned)iw >= (unsigned)W) continue;
        m = max(m, __ldg(xp + (int64_t)ih * W + iw));
      }
    }
    y[e] = m;
  }
}

// Max-pool 3x3, stride 2, padding 1 with W a multiple of 4 and OW = W / 2 even
// (every ResNet stem pool): a thread makes two neighbouring outputs of one row,
// reading per input row one 16-byte piece (columns 4q .. 4q+3) and the column
// before it, and stores the pair with one 8-byte store.
__global__ void maxpool3s2_pair_kernel(const int32_t* __restrict__ x, int32_t* __restrict__ y, int64_t planes,
                                       int H, int W, int OH, int OW, PoolIndex ix) {
  const int QW = OW / 2;
  const int64_t total = planes * OH * QW;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    int64_t pl;
    int oh, q;
    pool_coords(e, OH, QW, ix, pl, oh, q);
    const int32_t* xp = x + pl * H * W + 4 * q;
    int m0 = INT32_MIN, m1 = INT32_MIN;
#pragma unroll
    for (int r = 0; r < 3; ++r) {
      const int ih = 2 * oh - 1 + r;
      if ((unsigned)ih >= (unsigned)H) continue;
      const int4 v = __ldg(reinterpret_cast<const int4*>(xp + (int64_t)ih * W));
      const int left = q > 0 ? __ldg(xp + (int64_t)ih * W - 1) : INT32_MIN;
      m0 = max(m0, max(left, max(v.x, v.y)));
      m1 = max(m1, max(v.y, max(v.z, v.w)));
    }
    *reinterpret_cast<int2*>(y + (pl * OH + oh) * OW + 2 * q) = make_int2(m0, m1);
  }
}

// Average pool over whole planes (the global pool before a classifier): one
// warp per plane, lanes summing strided elements in 64 bits, then a shuffle
// reduction and the floor division.
__global__ void avgpool_plane_kernel(const int32_t* __restrict__ x, int32_t* __restrict__ y, int64_t planes,
                                     int HW) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t pl = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32; pl < planes; pl += warps) {
    const int32_t* xp = x + pl * HW;
    int64_t sum = 0;
    for (int i = lane; i < HW; i += 32) sum += __ldg(xp + i);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) {
      int64_t q = sum / HW;
      if (sum % HW != 0 && sum < 0) --q;  // floor
      y[pl] = (int32_t)q;
    }
  }
}

__global__ void avgpool_floor_kernel(const int32_t* __restrict__ x, int32_t* __restrict__ y, int64_t planes,
                                     int H, int W, int OH, int OW, int R, int S, int stride, PoolIndex ix) {
  const int64_t total = planes * OH * OW;
  const int64_t d = (int64_t)R * S;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    int64_t pl;
    int oh, ow;
    pool_coords(e, OH, OW, ix, pl, oh, ow);
    const int32_t* xp = x + pl * H * W + (int64_t)oh * stride * W + (int64_t)ow * stride;
    int64_t sum = 0;
    for (int r = 0; r < R; ++r)
      for (int s = 0; s < S; ++s) sum += __ldg(xp + (int64_t)r * W + s);
    int64_t q = sum / d;
    if (sum % d != 0 && sum < 0) --q;  // floor
    y[e] = (int32_t)q;
  }
}

static PoolIndex pool_index(int64_t planes, int OH, int OW) {
  const int64_t total = planes * OH * OW;
  return PoolIndex{make_fastdiv((uint32_t)OW), make_fastdiv((uint32_t)OH), total <= (int64_t)INT32_MAX};
}

static int64_t pool_blocks(int64_t total, int threads) {
  int64_t b = (total + threads - 1) / threads;
  const int64_t cap = (int64_t)(sm_count() > 0 ? sm_count() : 1) * 32;  // grid-stride beyond 32 CTAs per SM
  return b > cap ? cap : (b < 1 ? 1 : b);
}

cudaError_t launch_maxpool(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW, int R,
                           int S, int stride, int pad, cudaStream_t st) {
  const int threads = 256;
  if (R == 3 && S == 3 && stride == 2 && pad == 1 && W % 4 == 0 && 2 * OW == W &&
      (reinterpret_cast<uintptr_t>(x) & 15) == 0 && (reinterpret_cast<uintptr_t>(y) & 7) == 0) {
    maxpool3s2_pair_kernel<<<(unsigned)pool_blocks(planes * OH * (OW / 2), threads), threads, 0, st>>>(
        x, y, planes, H, W, OH, OW, pool_index(planes, OH, OW / 2));
    return cudaGetLastError();
  }
  maxpool_kernel<<<(unsigned)pool_blocks(planes * OH * OW, threads), threads, 0, st>>>(
      x, y, planes, H, W, OH, OW, R, S, stride, pad, pool_index(planes, OH, OW));
  return cudaGetLastError();
}

cudaError_t launch_avgpool_floor(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW,
                                 int R, int S, int stride, cudaStream_t st) {
  const int threads = 256;
  if (OH == 1 && OW == 1 && R == H && S == W && (int64_t)H * W <= (int64_t)INT32_MAX) {
    const int64_t blocks = std::min<int64_t>((planes + 7) / 8, (int64_t)(sm_count() > 0 ? sm_count() : 1) * 32);
    avgpool_plane_kernel<<<(unsigned)std::max<int64_t>(blocks, 1), threads, 0, st>>>(x, y, planes, H * W);
    return cudaGetLastError();
  }
  avgpool_floor_kernel<<<(unsigned)pool_blocks(planes * OH * OW, threads), threads, 0, st>>>(
      x, y, planes, H, W, OH, OW, R, S, stride, pool_index(planes, OH, OW));
  return cudaGetLastError();
}

}  // namespace ds
