// LinearShift and ConvShift forward kernels (DeepShift Eq. 1-3, Sec. 4).
//
// Both operators run as one integer "shift GEMM" on the CUDA cores:
//     y[row][col] = sat32( bias[col] + sum_k s[col][k] * (A[row][k] >> -p[col][k]) )
// with A = x for LinearShift and A = the implicit im2col matrix of x for
// ConvShift (rows = output pixels, k = (c, r, s), zero padding).
//
// Per term the hot loop issues exactly two instructions: an arithmetic right
// shift (ALU pipe) and an integer multiply-add by the sign s in {-1, 0, +1}
// (FMA pipe).  The two pipes issue in parallel, so the loop is bound by the
// SM's issue rate rather than by either pipe.  Codes are unpacked once per
// CTA tile into shared memory (shift and sign as 32-bit words), never per
// term, and the sign never branches.
//
// Accumulator width: 32-bit accumulation is used only when the launch-time
// bound  ceil(amax * A[col] / 2^15) + nnz[col] + |bias[col]| <= INT32_MAX
// holds for every column of the CTA tile (amax = max|x| from a pre-pass or
// the previous layer).  Then no wrap-around or saturation can occur and the
// 32-bit result is exact.  Otherwise the CTA runs the same loop with 64-bit
// accumulators and saturates the exact sum.
#include <algorithm>

#include "ds_common.cuh"

namespace ds {
namespace {

constexpr int MT = 128;       // rows per CTA tile
constexpr int NT = 64;        // columns per CTA tile
constexpr int TM = 8;         // rows per thread (rows tm + 16 i)
constexpr int TN = 8;         // columns per thread (cols tn * 8 + j)
constexpr int THREADS = 128;  // 16 row groups x 8 column groups
constexpr int XS = 36;        // words per x-tile row (32 + 4 pad: conflict-free 16 B reads)

struct __align__(16) Smem {
  int32_t xs[2][MT * XS];
  // codes per k: for each 32-column block, 32 shift amounts -p then 32 signs
  // (the expanded layout's row, so that layout is copied as is)
  int32_t cs[2][kChunk * 2 * NT];
};

// ---------------------------------------------------------------------------
// Staging of one 32-wide reduction chunk into a shared-memory stage.
// ---------------------------------------------------------------------------
struct RowCtx {
  // conv: the pixel this thread gathers for (one pixel per thread, MT == THREADS)
  int64_t img_base;  // n * C * H * W
  int ih0, iw0;      // oh * sh - ph, ow * sw - pw
  bool valid;
};

// FC x tile, 16-byte pieces: piece t + THREADS i is quad t % 8 of row
// t / 8 + 16 i, the same for every chunk, so the source address is computed
// once (row t / 8 at chunk 0) and the rows present kept as a bit mask.
struct XQuads {
  const int32_t* src;
  int64_t row_step;  // words between rows t / 8 + 16 i and t / 8 + 16 (i + 1)
  uint32_t rows_ok;  // bit i: row t / 8 + 16 i exists
};

__device__ __forceinline__ XQuads x_quads(const GemmParams& P, int64_t row0) {
  const int t = threadIdx.x;
  XQuads q;
  q.src = P.x + (row0 + (t >> 3)) * P.kred + 4 * (t & 7);
  q.row_step = 16 * P.kred;
  q.rows_ok = 0u;
#pragma unroll
  for (int i = 0; i < (MT * 8) / THREADS; ++i)
    if (row0 + (t >> 3) + 16 * i < P.rows) q.rows_ok |= 1u << i;
  return q;
}

template <bool CONV, bool VEC>
__device__ __forceinline__ void stage_x(const GemmParams& P, Smem& sm, int buf, int64_t row0,
                                        int64_t g, const RowCtx& rc, const XQuads& xq) {
  const int t = threadIdx.x;
  int32_t* xs = sm.xs[buf];
  if constexpr (!CONV) {
    if constexpr (VEC) {
      // 128 rows x 8 quads of 16 B; consecutive threads take consecutive quads.
      const bool k_ok = g * kChunk + 4 * (t & 7) < P.kred;
      const int32_t* src = xq.src + g * kChunk;
      int32_t* dst = xs + (t >> 3) * XS + 4 * (t & 7);
#pragma unroll
      for (int i = 0; i < (MT * 8) / THREADS; ++i) {
        const bool ok = k_ok && ((xq.rows_ok >> i) & 1u);
        cp_async16(dst + 16 * i * XS, ok ? src : P.x, ok);
        src += xq.row_step;
      }
    } else {
#pragma unroll 4
      for (int i = 0; i < (MT * kChunk) / THREADS; ++i) {
        const int e = t + THREADS * i;
        const int r = e >> 5, kk = e & 31;
        const int64_t row = row0 + r;
        const int64_t k = g * kChunk + kk;
        const bool ok = (row < P.rows) && (k < P.kred);
        const int32_t* src = ok ? (P.x + row * P.kred + k) : P.x;
        cp_async4(xs + r * XS + kk, src, ok);
      }
    }
  } else {
    // Implicit im2col: thread t gathers the 32 taps of chunk g for pixel t.
    const int RS = P.R * P.S;
    int64_t k = g * kChunk;
    int c = (int)(k / RS);
    int rem = (int)(k - (int64_t)c * RS);
    int r = rem / P.S;
    int s = rem - r * P.S;
    const int64_t HW = (int64_t)P.H * P.W;
    int32_t* dst = xs + t * XS;
#pragma unroll 4
    for (int kk = 0; kk < kChunk; ++kk) {
      const int ih = rc.ih0 + r, iw = rc.iw0 + s;
      const bool ok = rc.valid && (k + kk < P.kred) && ((unsigned)ih < (unsigned)P.H) &&
                      ((unsigned)iw < (unsigned)P.W);
      const int32_t* src = ok ? (P.x + rc.img_base + (int64_t)c * HW + (int64_t)ih * P.W + iw) : P.x;
      cp_async4(dst + kk, src, ok);
      if (++s == P.S) {
        s = 0;
        if (++r == P.R) {
          r = 0;
          ++c;
        }
      }
    }
  }
}

// Codes of chunk g for this CTA's columns: thread t owns column t % 64 and
// reduction half t / 64 (16 codes).  Loaded to registers first, decoded into
// shared memory later so the global latency overlaps the compute.
struct CodeRegs {
  uint2 nib;   // nibble words 2h, 2h+1
  uint2 bits;  // {sign, nz}
};

__device__ __forceinline__ CodeRegs load_codes(const GemmParams& P, int64_t col0, int64_t g) {
  const int t = threadIdx.x;
  const int64_t col = col0 + (t & (NT - 1));
  const int h = t >> 6;
  CodeRegs c;
  if (col < P.cols) {
    const int64_t rec = g * P.cols + col;
    c.nib = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_nib + rec * 16 + h * 8));
    c.bits = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
  } else {
    c.nib = make_uint2(0u, 0u);
    c.bits = make_uint2(0u, 0u);
  }
  return c;
}

__device__ __forceinline__ void store_codes(Smem& sm, int buf, const CodeRegs& c) {
  const int t = threadIdx.x;
  const int n = t & (NT - 1);
  const int h = t >> 6;
  int32_t* cs = sm.cs[buf] + (n >> 5) * 64 + (n & 31);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int k = 16 * h + i;
    const uint32_t w = (i < 8) ? c.nib.x : c.nib.y;
    const int sh = (int)((w >> (4 * (i & 7))) & 15u);
    const int neg = (int)((c.bits.x >> k) & 1u);
    const int nz = (int)((c.bits.y >> k) & 1u);
    cs[k * 2 * NT] = sh;
    cs[k * 2 * NT + 32] = nz - 2 * neg;
  }
}

// ---------------------------------------------------------------------------
// The hot loop over one staged chunk: 32 k x ROWS x 8 columns, two
// instructions per term (SHF + IMAD).
// ---------------------------------------------------------------------------
template <int ROW0, int ROWS, typename Acc>
__device__ __forceinline__ void compute_chunk(const Smem& sm, int buf, int tm, int tn,
                                              Acc (&acc)[ROWS][TN]) {
  const int32_t* xs = sm.xs[buf] + (tm + 16 * ROW0) * XS;
  static_assert(32 % TN == 0, "a thread's columns lie in one 32-column block");
  const int32_t* shs = sm.cs[buf] + ((tn * TN) >> 5) * 64 + ((tn * TN) & 31);
  const int32_t* sgs = shs + 32;
#pragma unroll 2
  for (int kq = 0; kq < kChunk / 4; ++kq) {
    int4 xv[ROWS];
#pragma unroll
    for (int i = 0; i < ROWS; ++i) xv[i] = *reinterpret_cast<const int4*>(xs + 16 * i * XS + 4 * kq);
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k = 4 * kq + kk;
      const int4 s0 = *reinterpret_cast<const int4*>(shs + k * 2 * NT);
      const int4 s1 = *reinterpret_cast<const int4*>(shs + k * 2 * NT + 4);
      const int4 g0 = *reinterpret_cast<const int4*>(sgs + k * 2 * NT);
      const int4 g1 = *reinterpret_cast<const int4*>(sgs + k * 2 * NT + 4);
      const int sh[TN] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
      const int sg[TN] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
      // column-outer order: consecutive SHF / IMAD share their shift / sign operand
#pragma unroll
      for (int j = 0; j < TN; ++j) {
#pragma unroll
        for (int i = 0; i < ROWS; ++i) {
          const int xk = kk == 0 ? xv[i].x : kk == 1 ? xv[i].y : kk == 2 ? xv[i].z : xv[i].w;
          const int t = xk >> sh[j];  // Eq. 1: arithmetic right shift by -p
          if constexpr (sizeof(Acc) == 4) {
            acc[i][j] += (uint32_t)sg[j] * (uint32_t)t;  // Eq. 2 flip + accumulate (mod 2^32)
          } else {
            acc[i][j] += (int64_t)sg[j] * (int64_t)t;
          }
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// One pass over the whole reduction for ROWS row slots starting at ROW0,
// then the fused epilogue (bias, saturation, residual, ReLU, amax).
// ---------------------------------------------------------------------------
template <bool CONV, bool VEC, int ROW0, int ROWS, typename Acc>
__device__ __forceinline__ void run_tile(const GemmParams& P, Smem& sm, int64_t row0, int64_t col0,
                                         const RowCtx& rc, uint32_t& amax_local) {
  const int t = threadIdx.x;
  const int tm = t & 15, tn = t >> 4;
  Acc acc[ROWS][TN];
#pragma unroll
  for (int i = 0; i < ROWS; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  const int64_t nch = P.n_chunks;
  // codes: the expanded layout is copied with cp.async next to x (two 16-index
  // halves per chunk); else decoded from the blob through registers, loaded
  // before the compute and stored after it
  const bool expanded = P.xcodes != nullptr;
  static_assert(THREADS == 128 && NT == 64 && kChunk == 32, "ExpandedCodeStager's stage shape, twice per chunk");
  const ExpandedCodeStager cst(P.xcodes, P.cols, P.kred, col0, 0);
  const XQuads xq = x_quads(P, row0);
  // prologue: chunk 0 into stage 0
  stage_x<CONV, VEC>(P, sm, 0, row0, 0, rc, xq);
  if (expanded) {
    cst.stage(P.xcodes, P.kred, sm.cs[0], 0);
    cst.stage(P.xcodes, P.kred, sm.cs[0] + 16 * 2 * NT, 1);
  }
  cp_async_commit();
  if (!expanded) {
    CodeRegs c0 = load_codes(P, col0, 0);
    store_codes(sm, 0, c0);
  }
  for (int64_t g = 0; g < nch; ++g) {
    const int buf = (int)(g & 1);
    const bool more = (g + 1 < nch);
    CodeRegs cn;
    if (more) {
      stage_x<CONV, VEC>(P, sm, buf ^ 1, row0, g + 1, rc, xq);
      if (expanded) {
        cst.stage(P.xcodes, P.kred, sm.cs[buf ^ 1], (int)(2 * g + 2));
        cst.stage(P.xcodes, P.kred, sm.cs[buf ^ 1] + 16 * 2 * NT, (int)(2 * g + 3));
      }
      cp_async_commit();
      if (!expanded) cn = load_codes(P, col0, g + 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    compute_chunk<ROW0, ROWS, Acc>(sm, buf, tm, tn, acc);
    if (more && !expanded) store_codes(sm, buf ^ 1, cn);
    __syncthreads();
  }

  // fused epilogue
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool resid = CONV && (P.flags & DS_RESIDUAL) != 0;
  int32_t bcol[TN];
#pragma unroll
  for (int j = 0; j < TN; ++j) {
    const int64_t col = col0 + tn * TN + j;
    bcol[j] = (P.bias != nullptr && col < P.cols) ? __ldg(P.bias + col) : 0;
  }
  const int64_t OHW = CONV ? (int64_t)P.OH * P.OW : 1;
#pragma unroll
  for (int i = 0; i < ROWS; ++i) {
    const int64_t row = row0 + tm + 16 * (ROW0 + i);
    if (row >= P.rows) continue;
    int32_t v[TN];
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      if constexpr (sizeof(Acc) == 4) {
        v[j] = (int32_t)(acc[i][j] + (uint32_t)bcol[j]);  // exact: the bound excludes overflow
      } else {
        int64_t a = acc[i][j] + (int64_t)bcol[j];
        a = a > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : a;
        a = a < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : a;
        v[j] = (int32_t)a;
      }
    }
    if constexpr (!CONV) {
      int32_t* yrow = P.y + row * P.cols + col0 + tn * TN;
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        if (relu) v[j] = max(v[j], 0);
        amax_local = max(amax_local, uabs(v[j]));
      }
      const int64_t cbase = col0 + tn * TN;
      if (cbase + TN <= P.cols && (P.cols & 3) == 0) {
        reinterpret_cast<int4*>(yrow)[0] = make_int4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<int4*>(yrow)[1] = make_int4(v[4], v[5], v[6], v[7]);
      } else {
#pragma unroll
        for (int j = 0; j < TN; ++j)
          if (cbase + j < P.cols) yrow[j] = v[j];
      }
    } else {
      const int64_t n = row / OHW;
      const int64_t pix = row - n * OHW;
      // output placement: pixel (oh, ow) of this grid -> (ys_h oh + yph, ys_w ow + ypw) of a yH x yW plane
      int64_t plane = OHW, off = pix;
      if (P.ys_h) {
        const int oh = (int)(pix / P.OW), ow = (int)(pix - (pix / P.OW) * P.OW);
        plane = (int64_t)P.yH * P.yW;
        off = (int64_t)(P.ys_h * oh + P.yph) * P.yW + P.ys_w * ow + P.ypw;
      }
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const int64_t col = col0 + tn * TN + j;
        if (col >= P.cols) continue;
        const int64_t idx = (n * P.cols + col) * plane + off;
        int32_t o = v[j];
        if (resid) o = add_sat(o, __ldg(P.residual + idx));
        if (relu) o = max(o, 0);
        amax_local = max(amax_local, uabs(o));
        P.y[idx] = o;
      }
    }
  }
}

// Whether 32-bit accumulation is exact for every column of this CTA tile.
__device__ __forceinline__ bool tile_int32_exact(const GemmParams& P, int64_t col0) {
  bool unsafe = false;
  const int t = threadIdx.x;
  if (P.amax_in == nullptr || (P.flags & DS_FORCE_INT64)) {
    unsafe = true;
  } else if (t < NT) {
    const int64_t col = col0 + t;
    if (col < P.cols) {
      const unsigned long long amax = *P.amax_in;
      const unsigned long long A = reinterpret_cast<const unsigned long long*>(P.blob + P.off_cola)[col];
      const unsigned long long nnz = reinterpret_cast<const uint32_t*>(P.blob + P.off_nnz)[col];
      const unsigned long long b = P.bias ? (unsigned long long)uabs(P.bias[col]) : 0ull;
      const unsigned long long hi = __umul64hi(amax, A);
      const unsigned long long lo = amax * A;
      if (hi != 0ull || lo > ~0ull - 32767ull) {
        unsafe = true;
      } else {
        const unsigned long long q = (lo + 32767ull) >> 15;
        unsafe = (q + nnz + b) > (unsigned long long)INT32_MAX;
      }
    }
  }
  return !__syncthreads_or(unsafe);
}

// One CTA tile (rows row0.., columns col0..) of the shift GEMM.
template <bool CONV, bool VEC>
__device__ __forceinline__ void gemm_cta(const GemmParams& P, Smem& sm, int64_t row0, int64_t col0) {
  RowCtx rc{0, 0, 0, false};
  if constexpr (CONV) {
    const int64_t pixel = row0 + threadIdx.x;
    rc.valid = pixel < P.rows;
    if (rc.valid) {
      const int64_t OHW = (int64_t)P.OH * P.OW;
      const int64_t n = pixel / OHW;
      const int pr = (int)(pixel - n * OHW);
      const int oh = pr / P.OW, ow = pr - (pr / P.OW) * P.OW;
      rc.img_base = n * (int64_t)P.C * P.H * P.W;
      rc.ih0 = oh * P.sh - P.ph;
      rc.iw0 = ow * P.sw - P.pw;
    }
  }

  uint32_t amax_local = 0;
  if (tile_int32_exact(P, col0)) {
    run_tile<CONV, VEC, 0, TM, uint32_t>(P, sm, row0, col0, rc, amax_local);
  } else {
    run_tile<CONV, VEC, 0, TM / 2, int64_t>(P, sm, row0, col0, rc, amax_local);
    run_tile<CONV, VEC, TM / 2, TM / 2, int64_t>(P, sm, row0, col0, rc, amax_local);
  }
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

template <bool CONV, bool VEC>
__global__ void __launch_bounds__(THREADS, 3) shift_gemm_kernel(const GemmParams P) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  gemm_cta<CONV, VEC>(P, *reinterpret_cast<Smem*>(smem_raw), (int64_t)blockIdx.x * MT, (int64_t)blockIdx.y * NT);
}

// Several implicit GEMMs in one launch (the tap phases of a strided layer's
// input gradient, each too small to fill the SMs alone): blockIdx.z picks the
// phase; a CTA beyond its phase's tiles returns at once.  The phases are
// selected by constant indices, so each reads its parameters at fixed offsets.
struct PhaseSet {
  GemmParams p[kMaxGemmPhases];
};

__device__ __forceinline__ void phase_cta(const GemmParams& P, Smem& sm) {
  const int64_t row0 = (int64_t)blockIdx.x * MT, col0 = (int64_t)blockIdx.y * NT;
  if (row0 >= P.rows || col0 >= P.cols) return;
  gemm_cta<true, false>(P, sm, row0, col0);
}

__global__ void __launch_bounds__(THREADS, 3) shift_gemm_phases_kernel(const PhaseSet S) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  switch (blockIdx.z) {
    case 0: phase_cta(S.p[0], sm); break;
    case 1: phase_cta(S.p[1], sm); break;
    case 2: phase_cta(S.p[2], sm); break;
    default: phase_cta(S.p[3], sm); break;
  }
}

template <bool CONV, bool VEC>
cudaError_t launch_impl(const GemmParams& p, cudaStream_t st) {
  const size_t smem = sizeof(Smem);
  // once per process, thread-safe (see conv_direct.cu)
  static const cudaError_t attr = cudaFuncSetAttribute(shift_gemm_kernel<CONV, VEC>,
                                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  dim3 grid((unsigned)((p.rows + MT - 1) / MT), (unsigned)((p.cols + NT - 1) / NT));
  shift_gemm_kernel<CONV, VEC><<<grid, THREADS, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_linear_shift(const GemmParams& p, cudaStream_t st) {
  const bool vec = (p.kred % 4 == 0) && ((reinterpret_cast<uintptr_t>(p.x) & 15) == 0);
  return vec ? launch_impl<false, true>(p, st) : launch_impl<false, false>(p, st);
}

cudaError_t launch_conv2d_shift(const GemmParams& p, cudaStream_t st) {
  return launch_impl<true, false>(p, st);
}

cudaError_t launch_conv2d_shift_phases(const GemmParams* ps, int n, cudaStream_t st) {
  static const cudaError_t attr = cudaFuncSetAttribute(shift_gemm_phases_kernel,
                                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                       (int)sizeof(Smem));
  if (attr != cudaSuccess) return attr;
  for (int i0 = 0; i0 < n; i0 += kMaxGemmPhases) {
    const int m = std::min(kMaxGemmPhases, n - i0);
    if (m == 1) {
      cudaError_t e = launch_conv2d_shift(ps[i0], st);
      if (e != cudaSuccess) return e;
      continue;
    }
    PhaseSet S{};
    int64_t rt = 0, ct = 0;
    for (int j = 0; j < m; ++j) {
      S.p[j] = ps[i0 + j];
      rt = std::max<int64_t>(rt, (ps[i0 + j].rows + MT - 1) / MT);
      ct = std::max<int64_t>(ct, (ps[i0 + j].cols + NT - 1) / NT);
    }
    shift_gemm_phases_kernel<<<dim3((unsigned)rt, (unsigned)ct, (unsigned)m), THREADS, sizeof(Smem), st>>>(S);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace ds
