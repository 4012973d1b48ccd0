// LinearShift for small batches: the reduction split over the CTAs of a
// thread-block cluster (DeepShift Eq. 1-3, Sec. 4).
//
//   y[m][n] = sat32( b[n] + sum_k s[n][k] * (x[m][k] >> -p[n][k]) )
//
// With few rows (a batch of 1 to a few hundred) the 128 x 64 tiles of
// shift_gemm.cu leave most SMs idle: a 64 x 784 x 512 layer makes 8 CTAs.
// Here a tile of MR = 8 * TMR rows x 64 columns belongs to one cluster of CS
// CTAs (CS <= 16, a power of two) along the reduction: CTA z of the cluster sums the terms of
// a 32-aligned slice of k.  Each CTA leaves its partial sums in its own shared
// memory; after a cluster barrier CTA z reduces one share of the tile over all
// CS partials through distributed shared memory (16-byte remote loads),
// applies the epilogue (bias, saturation, ReLU, max|y|) and stores; a second
// cluster barrier keeps every CTA's shared memory alive until the remote
// reads are done.  No global scratch memory is used.
//
// 128 threads: thread (tm, tn) = (t % 8, t / 8) owns rows tm + 8 i (i < TMR)
// and columns 4 tn .. 4 tn + 3.  Per reduction chunk of 32 k the CTA stages
// x rows (16-byte cp.async when K % 4 == 0) and the chunk's codes (expanded
// layout: 16-byte cp.async; else decoded from the packed blob).  Per term the
// hot loop is one SHF and one IMAD, as in shift_gemm.cu.  Accumulator width
// as in shift_gemm.cu: the bound proven for the whole sum also covers every
// partial sum (a subset of its terms), so 32-bit partials are exact whenever
// the 32-bit path is taken, and their wrap-around sum is the exact sum.
#include <cooperative_groups.h>

#include <algorithm>

#include "ds_common.cuh"

namespace cg = cooperative_groups;

namespace ds {
namespace {

constexpr int NT = 64;        // columns per tile
constexpr int TN = 4;         // columns per thread
constexpr int THREADS = 128;  // 8 row groups x 16 column groups
constexpr int KC = kChunk;    // reduction indices per stage (one packed chunk)
constexpr int XS = KC + 4;    // words per staged x row (16-byte reads of 8 rows hit distinct banks)
constexpr int CW = 2 * 64;    // code words per k: 2 blocks of {32 shifts, 32 signs}
constexpr int kSlots = 152 * 4;  // resident CTAs on a GB300 at 4 per SM
constexpr int kMaxCluster = 16;

template <int TMR>
struct ClSmem {
  static constexpr int MR = 8 * TMR;
  int32_t xs[2][MR * XS];
  int32_t cs[2][KC * CW];
};

__device__ __forceinline__ void cp_async4(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(gsrc), "r"(valid ? 4 : 0));
}
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(gsrc), "r"(valid ? 16 : 0));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::); }
__device__ __forceinline__ uint32_t uabs(int32_t v) { return v < 0 ? (uint32_t)0 - (uint32_t)v : (uint32_t)v; }

// x rows [row0, row0 + MR), reduction indices [k0, k0 + 32) clipped to kend
// (the end of this CTA's slice); zero elsewhere.
template <int TMR, bool VEC>
__device__ __forceinline__ void stage_x(const GemmParams& P, int32_t* xs, int64_t row0, int64_t k0, int64_t kend) {
  constexpr int MR = 8 * TMR;
  if constexpr (VEC) {
    for (int e = threadIdx.x; e < MR * (KC / 4); e += THREADS) {
      const int r = e / (KC / 4), q = e % (KC / 4);
      const int64_t row = row0 + r, k = k0 + 4 * q;
      const bool ok = row < P.rows && k < kend;  // K % 4 == 0 and kend is 32-aligned or K: whole pieces
      cp_async16(xs + r * XS + 4 * q, ok ? (const void*)(P.x + row * P.kred + k) : (const void*)P.x, ok);
    }
  } else {
    for (int e = threadIdx.x; e < MR * KC; e += THREADS) {
      const int r = e / KC, kk = e % KC;
      const int64_t row = row0 + r, k = k0 + kk;
      const bool ok = row < P.rows && k < kend;
      cp_async4(xs + r * XS + kk, ok ? (const void*)(P.x + row * P.kred + k) : (const void*)P.x, ok);
    }
  }
}

// Codes of chunk k0 / 32 for columns [col0, col0 + 64) from the expanded layout.
__device__ __forceinline__ void stage_codes_expanded(const GemmParams& P, int32_t* cs, int64_t col0, int64_t k0) {
  const int64_t nblocks = (P.cols + 31) / 32;
  for (int e = threadIdx.x; e < 2 * KC * 16; e += THREADS) {
    const int b = e / (KC * 16);
    const int r = e - b * KC * 16;
    const int kl = r >> 4, q = r & 15;
    const int64_t cb = col0 / 32 + b;
    const bool ok = cb < nblocks && k0 + kl < P.kred;
    const int32_t* src = ok ? P.xcodes + ((cb * P.kred + k0 + kl) * 64 + q * 4) : P.xcodes;
    cp_async16(cs + kl * CW + b * 64 + q * 4, src, ok);
  }
}

// Blob path: thread t decodes 16 indices (half t / 64) of column t % 64 of
// chunk g (indices past k_red decode to s = 0: the blob's padding is zero).
__device__ __forceinline__ void decode_codes(const GemmParams& P, int32_t* cs, int64_t col0, int64_t g) {
  const int t = threadIdx.x;
  const int n = t & 63;
  const int h = t >> 6;
  const int64_t col = col0 + n;
  uint2 nib = make_uint2(0u, 0u), bits = make_uint2(0u, 0u);
  if (col < P.cols) {
    const int64_t rec = g * P.cols + col;
    nib = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_nib + rec * 16 + h * 8));
    bits = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
  }
  int32_t* base = cs + (n >> 5) * 64 + (n & 31);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int k = 16 * h + i;
    const uint32_t w = i < 8 ? nib.x : nib.y;
    base[k * CW] = (int)((w >> (4 * (i & 7))) & 15u);
    base[k * CW + 32] = (int)((bits.y >> k) & 1u) - 2 * (int)((bits.x >> k) & 1u);
  }
}

template <int TMR, typename Acc>
__device__ __forceinline__ void compute_chunk(const int32_t* xs, const int32_t* cs, int tm, int tn,
                                              Acc (&acc)[TMR][TN]) {
  const int32_t* cb = cs + ((tn * TN) >> 5) * 64 + ((tn * TN) & 31);
#pragma unroll 2
  for (int k4 = 0; k4 < KC / 4; ++k4) {
    int4 xv[TMR];
#pragma unroll
    for (int i = 0; i < TMR; ++i) xv[i] = *reinterpret_cast<const int4*>(xs + (tm + 8 * i) * XS + 4 * k4);
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k = 4 * k4 + kk;
      const int4 s4 = *reinterpret_cast<const int4*>(cb + k * CW);
      const int4 g4 = *reinterpret_cast<const int4*>(cb + k * CW + 32);
      const int sh[TN] = {s4.x, s4.y, s4.z, s4.w};
      const int sg[TN] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
      for (int i = 0; i < TMR; ++i) {
        const int x = kk == 0 ? xv[i].x : kk == 1 ? xv[i].y : kk == 2 ? xv[i].z : xv[i].w;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
          const int t = x >> sh[j];  // Eq. 1
          if constexpr (sizeof(Acc) == 4) {
            acc[i][j] += (uint32_t)sg[j] * (uint32_t)t;  // Eq. 2 + accumulate (mod 2^32)
          } else {
            acc[i][j] += (int64_t)sg[j] * (int64_t)t;
          }
        }
      }
    }
  }
}

// Whether 32-bit accumulation is exact for every column of the tile (the
// bound of shift_gemm.cu).  The same for every CTA of a cluster.
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
      unsafe = (hi != 0ull || lo > ~0ull - 32767ull) ? true
                                                     : (((lo + 32767ull) >> 15) + nnz + b) > (unsigned long long)INT32_MAX;
    }
  }
  return !__syncthreads_or(unsafe);
}

template <int TMR, bool VEC, typename Acc>
__device__ __forceinline__ void run_cluster_tile(const GemmParams& P, ClSmem<TMR>& sm, cg::cluster_group& cl,
                                                 int64_t row0, int64_t col0, int64_t kbeg, int64_t kend,
                                                 uint32_t& amax_local) {
  constexpr int MR = 8 * TMR;
  const int t = threadIdx.x;
  const int tm = t % 8, tn = t / 8;
  const bool expanded = P.xcodes != nullptr;
  Acc acc[TMR][TN];
#pragma unroll
  for (int i = 0; i < TMR; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  // a trailing CTA of the cluster may have an empty slice: it stages nothing
  // and contributes zero partial sums
  const int nst = kend > kbeg ? (int)((kend - kbeg + KC - 1) / KC) : 0;
  if (nst > 0) {
    stage_x<TMR, VEC>(P, sm.xs[0], row0, kbeg, kend);
    if (expanded) stage_codes_expanded(P, sm.cs[0], col0, kbeg);
    cp_async_commit();
    if (!expanded) decode_codes(P, sm.cs[0], col0, kbeg / KC);
    cp_async_wait_all();
  }
  for (int st = 0; st < nst; ++st) {
    const int b = st & 1;
    const bool more = st + 1 < nst;
    const int64_t k1 = kbeg + (int64_t)(st + 1) * KC;
    __syncthreads();
    if (more) {
      stage_x<TMR, VEC>(P, sm.xs[b ^ 1], row0, k1, kend);
      if (expanded) stage_codes_expanded(P, sm.cs[b ^ 1], col0, k1);
      cp_async_commit();
    }
    compute_chunk<TMR, Acc>(sm.xs[b], sm.cs[b], tm, tn, acc);
    if (more) {
      if (!expanded) decode_codes(P, sm.cs[b ^ 1], col0, k1 / KC);
      cp_async_wait_all();
    }
  }
  __syncthreads();  // every thread is done with the staging buffers: they hold the partials next

  // this CTA's partial sums, [MR][64] row-major, 16 bytes per (row, 4 columns) for 32-bit
  Acc* red = reinterpret_cast<Acc*>(&sm);
#pragma unroll
  for (int i = 0; i < TMR; ++i) {
    Acc* dst = red + (tm + 8 * i) * NT + tn * TN;
#pragma unroll
    for (int j = 0; j < TN; ++j) dst[j] = acc[i][j];
  }
  cl.sync();  // all partials of the cluster are written and visible

  const int rank = (int)cl.block_rank();
  const int cs_n = (int)cl.num_blocks();
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool vec_out = (P.cols % 4) == 0;
  constexpr int GROUPS = MR * (NT / TN);  // (row, 4 columns) groups of the tile
  for (int gi = rank * THREADS + t; gi < GROUPS; gi += cs_n * THREADS) {
    const int r = gi / (NT / TN), c4 = gi % (NT / TN);
    Acc sum[TN] = {0, 0, 0, 0};
    for (int q = 0; q < cs_n; ++q) {
      const Acc* src = cl.map_shared_rank(red, q) + r * NT + c4 * TN;
      if constexpr (sizeof(Acc) == 4) {
        const uint4 v = *reinterpret_cast<const uint4*>(src);
        sum[0] += v.x;
        sum[1] += v.y;
        sum[2] += v.z;
        sum[3] += v.w;
      } else {
        const longlong2 v0 = *reinterpret_cast<const longlong2*>(src);
        const longlong2 v1 = *reinterpret_cast<const longlong2*>(src + 2);
        sum[0] += v0.x;
        sum[1] += v0.y;
        sum[2] += v1.x;
        sum[3] += v1.y;
      }
    }
    const int64_t row = row0 + r;
    if (row >= P.rows) continue;
    const int64_t col = col0 + c4 * TN;
    int32_t o[TN];
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int32_t b = (P.bias != nullptr && col + j < P.cols) ? __ldg(P.bias + col + j) : 0;
      if constexpr (sizeof(Acc) == 4) {
        o[j] = (int32_t)(sum[j] + (uint32_t)b);
      } else {
        int64_t v = sum[j] + (int64_t)b;
        v = v > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : v;
        v = v < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : v;
        o[j] = (int32_t)v;
      }
      if (relu) o[j] = max(o[j], 0);
    }
    int32_t* yp = P.y + row * P.cols + col;
    if (vec_out && col + TN <= P.cols) {
#pragma unroll
      for (int j = 0; j < TN; ++j) amax_local = max(amax_local, uabs(o[j]));
      *reinterpret_cast<int4*>(yp) = make_int4(o[0], o[1], o[2], o[3]);
    } else {
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        if (col + j < P.cols) {
          amax_local = max(amax_local, uabs(o[j]));
          yp[j] = o[j];
        }
      }
    }
  }
  cl.sync();  // no CTA leaves (or reuses its shared memory) while another still reads it
}

template <int TMR, bool VEC>
__global__ void __launch_bounds__(THREADS, 4) linear_cluster_kernel(const GemmParams P, int64_t k_per_cta) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  ClSmem<TMR>& sm = *reinterpret_cast<ClSmem<TMR>*>(smem_raw);
  cg::cluster_group cl = cg::this_cluster();
  const int64_t row0 = (int64_t)blockIdx.x * (8 * TMR);
  const int64_t col0 = (int64_t)blockIdx.y * NT;
  const int64_t kbeg = (int64_t)cl.block_rank() * k_per_cta;
  const int64_t kend = min(P.kred, kbeg + k_per_cta);
  uint32_t amax_local = 0;
  if (tile_int32_exact(P, col0)) {
    run_cluster_tile<TMR, VEC, uint32_t>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
  } else {
    run_cluster_tile<TMR, VEC, int64_t>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
  }
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

// Largest cluster size (<= 16) the device can co-schedule for this kernel,
// queried once per process.
template <int TMR, bool VEC>
cudaError_t prepare(size_t smem, int& max_cluster) {
  static int cached = 0;
  if (cached > 0) {
    max_cluster = cached;
    return cudaSuccess;
  }
  auto kern = linear_cluster_kernel<TMR, VEC>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  int best = 1;
  for (int cs = kMaxCluster; cs >= 2; cs /= 2) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1, 1, cs);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = cs;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n > 0) {
      best = cs;
      break;
    }
    (void)cudaGetLastError();  // clear a refused query
  }
  cached = best;
  max_cluster = best;
  return cudaSuccess;
}

template <int TMR, bool VEC>
cudaError_t launch_tmr(const GemmParams& p, cudaStream_t st) {
  constexpr int MR = 8 * TMR;
  const size_t smem = sizeof(ClSmem<TMR>);
  static_assert(sizeof(ClSmem<TMR>) >= (size_t)MR * NT * sizeof(int64_t), "partials fit the staging buffers");
  int max_cluster = 1;
  cudaError_t e = prepare<TMR, VEC>(smem, max_cluster);
  if (e != cudaSuccess) return e;
  const int64_t tiles = ((p.rows + MR - 1) / MR) * ((p.cols + NT - 1) / NT);
  const int64_t chunks = (p.kred + KC - 1) / KC;
  // the cluster size: a power of two that fills at most one wave of CTAs and
  // gives every CTA at least one chunk (trailing slices may still be empty)
  const int64_t want = std::min<int64_t>(std::min<int64_t>(kSlots / std::max<int64_t>(tiles, 1), max_cluster), chunks);
  int64_t cs = 1;
  while (cs * 2 <= want) cs *= 2;
  const int64_t chunks_per_cta = (chunks + cs - 1) / cs;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((p.rows + MR - 1) / MR), (unsigned)((p.cols + NT - 1) / NT), (unsigned)cs);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 1;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = (unsigned)cs;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, linear_cluster_kernel<TMR, VEC>, p, chunks_per_cta * KC);
}

template <bool VEC>
cudaError_t launch_by_rows(const GemmParams& p, cudaStream_t st) {
  if (p.rows <= 8) return launch_tmr<1, VEC>(p, st);
  if (p.rows <= 32) return launch_tmr<4, VEC>(p, st);
  return launch_tmr<8, VEC>(p, st);
}

}  // namespace

bool linear_cluster_preferred(const GemmParams& p) {
  // the 128 x 64 tiles of shift_gemm.cu would not fill the SMs three times over
  const int64_t gemm_ctas = ((p.rows + 127) / 128) * ((p.cols + NT - 1) / NT);
  return gemm_ctas < 3 * 152 && (p.cols + NT - 1) / NT <= 65535 && (p.rows + 7) / 8 <= (int64_t)INT32_MAX;
}

cudaError_t launch_linear_cluster(const GemmParams& p, cudaStream_t st) {
  const bool vec = (p.kred % 4 == 0) && ((reinterpret_cast<uintptr_t>(p.x) & 15) == 0);
  return vec ? launch_by_rows<true>(p, st) : launch_by_rows<false>(p, st);
}

}  // namespace ds
