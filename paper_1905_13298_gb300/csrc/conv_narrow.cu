// ConvShift with few output columns (DeepShift Eq. 1-3, Sec. 4): the
// input-gradient phases of a layer whose input has few channels (Eq. 7: the
// gradient of a ResNet stem has C = 3 columns), where the 64-column tiles of
// the implicit GEMM would leave most of their columns empty.
//
//   y[row][col] = sat32( bias[col] + sum_{c,r,s} s_w * (xpad[n][c][oh + r][ow + s] >> -p) ),  stride 1
//
// A thread owns TP = 4 consecutive output pixels of one row and all NC (4 or
// 8) columns.  Per (c, r) it loads the TP + S - 1 input values of its row
// once (L1-cached global loads, zero outside the image) and reuses them for
// the S taps; per tap the CTA's codes for the NC columns come from shared
// memory as broadcast 16-byte loads, and each term is one shift (ALU pipe)
// and one multiply-add by the sign (FMA pipe).  The codes of a run of input
// channels are staged once per CTA (copied from the expanded layout, or
// decoded from the packed blob).  Output placement, bias, residual, ReLU,
// saturation and max|y| as in the implicit GEMM (shift_gemm.cu); the
// accumulator width is proven per CTA in the same way.
#include <algorithm>

#include "ds_common.cuh"

namespace ds {
namespace {

constexpr int TP = 4;           // output pixels per thread (one row)
constexpr int THREADS = 128;
constexpr int kCodeWords = 8192;  // shared-memory words for staged codes (32 KB)

template <int NC>
__device__ __forceinline__ void stage_codes(const GemmParams& P, int32_t* cs, int64_t k0, int nk) {
  // cs[k][0..NC) = -p, cs[k][NC..2NC) = s of the columns (zero beyond cols)
  if (P.xcodes != nullptr) {
    // the expanded layout's row of k holds the NC columns' shifts and signs contiguously (zero beyond
    // n_out): 16-byte loads, several in flight per thread
#pragma unroll 4
    for (int kk = threadIdx.x; kk < nk; kk += THREADS) {
      const int4* src = reinterpret_cast<const int4*>(P.xcodes + (k0 + kk) * 64);
      int4* dst = reinterpret_cast<int4*>(cs + kk * 2 * NC);
#pragma unroll
      for (int v = 0; v < NC / 4; ++v) {
        dst[v] = __ldg(src + v);
        dst[NC / 4 + v] = __ldg(src + 8 + v);
      }
    }
    return;
  }
  for (int i = threadIdx.x; i < nk * NC; i += THREADS) {
    const int kk = i / NC, col = i - kk * NC;
    const int64_t k = k0 + kk;
    int sh = 0, sg = 0;
    if (col < P.cols) {
      const int64_t g = k >> 5;
      const int j = (int)(k & 31);
      const uint32_t nib =
          __ldg(reinterpret_cast<const uint32_t*>(P.blob + P.off_nib) + (g * P.cols + col) * 4 + (j >> 3));
      const uint2 bits = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits) + g * P.cols + col);
      sh = (int)((nib >> (4 * (j & 7))) & 15u);
      sg = ((bits.y >> j) & 1u) ? (((bits.x >> j) & 1u) ? -1 : 1) : 0;
    }
    cs[kk * 2 * NC + col] = sh;
    cs[kk * 2 * NC + NC + col] = sg;
  }
}

// Whether 32-bit accumulation is exact for every column (the bound of shift_gemm.cu).
__device__ __forceinline__ bool narrow_int32_exact(const GemmParams& P) {
  bool unsafe = false;
  const int t = threadIdx.x;
  if (P.amax_in == nullptr || (P.flags & DS_FORCE_INT64)) {
    unsafe = true;
  } else if (t < P.cols) {
    const unsigned long long amax = *P.amax_in;
    const unsigned long long A = reinterpret_cast<const unsigned long long*>(P.blob + P.off_cola)[t];
    const unsigned long long nnz = reinterpret_cast<const uint32_t*>(P.blob + P.off_nnz)[t];
    const unsigned long long b = P.bias ? (unsigned long long)uabs(P.bias[t]) : 0ull;
    const unsigned long long hi = __umul64hi(amax, A);
    const unsigned long long lo = amax * A;
    if (hi != 0ull || lo > ~0ull - 32767ull)
      unsafe = true;
    else
      unsafe = (((lo + 32767ull) >> 15) + nnz + b) > (unsigned long long)INT32_MAX;
  }
  return !__syncthreads_or(unsafe);
}

// The TP + S - 1 input values of one row segment (zero outside the image).
template <int S>
__device__ __forceinline__ void load_row(const GemmParams& P, const int32_t* xc, int ih, int iw0, int* w) {
  const bool row_ok = (unsigned)ih < (unsigned)P.H;
  const int32_t* xr = xc + (int64_t)(row_ok ? ih : 0) * P.W;
#pragma unroll
  for (int i = 0; i < TP + S - 1; ++i) {
    const int iw = iw0 + i;
    w[i] = (row_ok && (unsigned)iw < (unsigned)P.W) ? __ldg(xr + iw) : 0;
  }
}

// The S taps of one (c, r) row: codes ck[s][0..NC) = -p, ck[s][NC..2NC) = s.
template <int NC, int S, typename Acc>
__device__ __forceinline__ void row_terms(const int32_t* ck, const int* w, Acc (&acc)[TP][NC]) {
#pragma unroll
  for (int s = 0; s < S; ++s) {
    int sh[NC], sg[NC];
#pragma unroll
    for (int v = 0; v < NC / 4; ++v) {
      const int4 a = reinterpret_cast<const int4*>(ck + s * 2 * NC)[v];
      const int4 b = reinterpret_cast<const int4*>(ck + s * 2 * NC + NC)[v];
      sh[4 * v] = a.x, sh[4 * v + 1] = a.y, sh[4 * v + 2] = a.z, sh[4 * v + 3] = a.w;
      sg[4 * v] = b.x, sg[4 * v + 1] = b.y, sg[4 * v + 2] = b.z, sg[4 * v + 3] = b.w;
    }
#pragma unroll
    for (int j = 0; j < NC; ++j)
#pragma unroll
      for (int t = 0; t < TP; ++t) acc[t][j] += (Acc)sg[j] * (Acc)(w[t + s] >> sh[j]);
  }
}

template <int NC, int S, typename Acc>
__device__ __forceinline__ void run_narrow(const GemmParams& P, int32_t* cs, int ch_per_run, uint32_t& amax_local) {
  const int OWQ = (P.OW + TP - 1) / TP;
  const int64_t quads = (int64_t)(P.rows / ((int64_t)P.OH * P.OW)) * P.OH * OWQ;
  const int64_t q = (int64_t)blockIdx.x * THREADS + threadIdx.x;
  const bool active = q < quads;
  int64_t n = 0;
  int oh = 0, ow0 = 0;
  if (active) {
    const int64_t nr = q / OWQ;
    ow0 = (int)(q - nr * OWQ) * TP;
    n = nr / P.OH;
    oh = (int)(nr - n * P.OH);
  }
  Acc acc[TP][NC];
#pragma unroll
  for (int t = 0; t < TP; ++t)
#pragma unroll
    for (int j = 0; j < NC; ++j) acc[t][j] = 0;
  const int64_t HW = (int64_t)P.H * P.W;
  const int iw0 = ow0 - P.pw;
  for (int c0 = 0; c0 < P.C; c0 += ch_per_run) {
    const int nc = min(ch_per_run, P.C - c0);
    __syncthreads();  // the previous run's codes are no longer read
    stage_codes<NC>(P, cs, (int64_t)c0 * P.R * S, nc * P.R * S);
    __syncthreads();
    const int32_t* xc0 = P.x + (n * P.C + c0) * HW;
    if (!active) continue;
    // the (c, r) rows of the run in order, the next row's input values loaded while the current row's terms run
    const int rows = nc * P.R;
    int w0[TP + S - 1], w1[TP + S - 1];
    load_row<S>(P, xc0 + 0, oh - P.ph, iw0, w0);
    for (int it = 0; it < rows; it += 2) {
      const int c1 = (it + 1) / P.R, r1 = it + 1 - c1 * P.R;
      if (it + 1 < rows) load_row<S>(P, xc0 + c1 * HW, oh + r1 - P.ph, iw0, w1);
      row_terms<NC, S>(cs + it * S * 2 * NC, w0, acc);
      if (it + 1 < rows) {
        if (it + 2 < rows) {
          const int c2 = (it + 2) / P.R, r2 = it + 2 - c2 * P.R;
          load_row<S>(P, xc0 + c2 * HW, oh + r2 - P.ph, iw0, w0);
        }
        row_terms<NC, S>(cs + (it + 1) * S * 2 * NC, w1, acc);
      }
    }
  }
  if (!active) return;
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool resid = (P.flags & DS_RESIDUAL) != 0 && P.residual != nullptr;
  int64_t plane = (int64_t)P.OH * P.OW;
  if (P.ys_h) plane = (int64_t)P.yH * P.yW;
#pragma unroll
  for (int t = 0; t < TP; ++t) {
    const int ow = ow0 + t;
    if (ow >= P.OW) break;
    const int64_t off = P.ys_h ? (int64_t)(P.ys_h * oh + P.yph) * P.yW + P.ys_w * ow + P.ypw
                               : (int64_t)oh * P.OW + ow;
#pragma unroll
    for (int j = 0; j < NC; ++j) {
      if (j >= P.cols) break;
      const int64_t idx = (n * P.cols + j) * plane + off;
      int32_t o;
      if constexpr (sizeof(Acc) == 4) {
        o = (int32_t)((uint32_t)acc[t][j] + (uint32_t)(P.bias ? P.bias[j] : 0));
      } else {
        int64_t v = (int64_t)acc[t][j] + (P.bias ? (int64_t)P.bias[j] : 0);
        v = v > INT32_MAX ? INT32_MAX : (v < INT32_MIN ? INT32_MIN : v);
        o = (int32_t)v;
      }
      if (resid) o = add_sat(o, __ldg(P.residual + idx));
      if (relu) o = max(o, 0);
      amax_local = max(amax_local, uabs(o));
      P.y[idx] = o;
    }
  }
}

template <int NC, int S>
__global__ void __launch_bounds__(THREADS, 4) conv_narrow_kernel(const GemmParams P, int ch_per_run) {
  __shared__ __align__(16) int32_t cs[kCodeWords];
  uint32_t amax_local = 0;
  if (narrow_int32_exact(P))
    run_narrow<NC, S, uint32_t>(P, cs, ch_per_run, amax_local);
  else
    run_narrow<NC, S, int64_t>(P, cs, ch_per_run, amax_local);
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

template <int NC, int S>
cudaError_t launch_s(const GemmParams& p, cudaStream_t st) {
  const int per_c = p.R * S * 2 * NC;
  const int ch_per_run = std::max(1, std::min(p.C, kCodeWords / per_c));
  const int64_t quads = (p.rows / ((int64_t)p.OH * p.OW)) * p.OH * ((p.OW + TP - 1) / TP);
  const int64_t blocks = (quads + THREADS - 1) / THREADS;
  conv_narrow_kernel<NC, S><<<(unsigned)blocks, THREADS, 0, st>>>(p, ch_per_run);
  return cudaGetLastError();
}

template <int NC>
cudaError_t launch_nc(const GemmParams& p, cudaStream_t st) {
  switch (p.S) {
    case 1: return launch_s<NC, 1>(p, st);
    case 2: return launch_s<NC, 2>(p, st);
    case 3: return launch_s<NC, 3>(p, st);
    default: return launch_s<NC, 4>(p, st);
  }
}

}  // namespace

bool conv_narrow_supported(const GemmParams& p) {
  return p.cols >= 1 && p.cols <= 8 && p.sh == 1 && p.sw == 1 && p.S >= 1 && p.S <= 4 && p.R >= 1 &&
         p.R * p.S * 2 * 8 <= kCodeWords && p.split_acc == nullptr &&
         (p.rows / ((int64_t)p.OH * p.OW)) * p.OH * ((p.OW + TP - 1) / TP) <= (int64_t)INT32_MAX * THREADS;
}

cudaError_t launch_conv_narrow(const GemmParams& p, cudaStream_t st) {
  return p.cols <= 4 ? launch_nc<4>(p, st) : launch_nc<8>(p, st);
}

}  // namespace ds
