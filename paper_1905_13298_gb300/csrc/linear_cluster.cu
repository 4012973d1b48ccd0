// LinearShift for small batches: the reduction split over the CTAs of a
// thread-block cluster (DeepShift Eq. 1-3, Sec. 4).
//
//   y[m][n] = sat32( b[n] + sum_k s[n][k] * (x[m][k] >> -p[n][k]) )
//
// With few rows (a batch of 1 to a few hundred) the 128 x 64 tiles of
// shift_gemm.cu leave most SMs idle: a 64 x 784 x 512 layer makes 8 CTAs.
// Here a tile of MR = 8 * TMR rows x 64 columns belongs to one cluster of CS
// CTAs (CS <= 16) along the reduction: CTA z of the cluster sums the terms of
// a 16-aligned slice of k.  Each CTA leaves its partial sums in its own shared
// memory; after a cluster barrier CTA z reduces one share of the tile over all
// CS partials through distributed shared memory (16-byte remote loads),
// applies the epilogue (bias, saturation, ReLU, max|y|) and stores; a second
// cluster barrier keeps every CTA's shared memory alive until the remote
// reads are done.  No global scratch memory is used.
//
// 128 threads: thread (tm, tn) = (t % 8, t / 8) owns columns 4 tn .. 4 tn + 3
// and TMR rows: row tm (TMR = 1), rows 4 tm .. 4 tm + 3 (TMR = 4), or two such
// quads 32 rows apart (TMR = 8), so that the 8 row groups of a warp read
// distinct banks.  Per stage of 16 k the CTA stages x transposed ([k][row], so
// a thread's rows at one k are one or two 16-byte loads) and the stage's
// codes (expanded layout: 16-byte cp.async; else decoded from the packed
// blob; the expanded copy is ExpandedCodeStager).  x arrives in 16-byte pieces of 4 k of one row (4-byte copies when K
// is not a multiple of 4, as rows are then not 16-byte aligned) in a row-major
// scratch tile; once a thread's own copies have landed it writes its pieces
// transposed, so no barrier is added.  Every thread copies the same pieces at
// every stage: its source pointers only advance by 16 k.  Per term the hot
// loop is one SHF and one IMAD, as in shift_gemm.cu; at most 96 registers,
// 5 CTAs per SM.
// Accumulator width as in shift_gemm.cu: the bound proven for the whole sum
// also covers every partial sum (a subset of its terms), so 32-bit partials
// are exact whenever the 32-bit path is taken, and their wrap-around sum is
// the exact sum.
#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>

#include "ds_common.cuh"

namespace cg = cooperative_groups;

namespace ds {
namespace {

constexpr int NT = 64;        // columns per tile
constexpr int TN = 4;         // columns per thread
constexpr int THREADS = 128;  // 8 row groups x 16 column groups
constexpr int KC = 16;        // reduction indices per stage (half of a packed 32-index chunk)
constexpr int CW = 2 * 64;    // code words per k: 2 blocks of {32 shifts, 32 signs}
constexpr int kMinBlocks = 5;
// resident CTAs of the device (kMinBlocks per SM)
inline int64_t slots() { return (int64_t)sm_count() * kMinBlocks; }
constexpr int kMaxCluster = 16;

template <int TMR>
struct ClSmem {
  static constexpr int MR = 8 * TMR;
  static constexpr int XR = MR + 4;  // words per staged k (16-byte aligned rows of the transposed tile)
  union {
    struct {
      int32_t xs[2][KC * XR];
      int32_t cs[2][KC * CW];
      int32_t xt[MR * KC];  // x of the stage in flight, row-major [row][16 k]
    } st;
    int64_t red[MR * NT];  // the partial sums (int64 or int32) after the reduction loop
  };
};

// x rows [row0, row0 + MR), reduction indices [k0, k0 + 16) clipped to kend
// (the end of this CTA's slice); zero elsewhere.  Piece e of a stage (e =
// threadIdx.x + THREADS u) is 4 consecutive k of one row: with 32 rows or
// more, a warp's pieces are 16 consecutive rows x 2 adjacent pieces (each
// row's 32 bytes read together, and the transposing 4-byte stores of the two
// halves of the warp fall on the two halves of the banks); with 8 rows, row
// e / 4, piece e % 4.  copy() puts a piece at xt[4 e] (XV: one 16-byte copy
// whose source size zero-fills a ragged end; else four 4-byte copies),
// transpose() moves the thread's own landed pieces to xs[k][row].  src[u]:
// the piece's address at stage 0.
template <int TMR, bool XV>
struct XStager {
  static constexpr int MR = 8 * TMR;
  static constexpr int NP = MR * KC / 4;                       // pieces per stage
  static constexpr int PIECES = (NP + THREADS - 1) / THREADS;  // per thread: 1, 1, 2
  const int32_t* src[PIECES];
  int64_t kp[PIECES];  // the piece's first k at stage 0, or the slice end if its row is absent
  __device__ __forceinline__ static int piece_row(int e) {
    if constexpr (MR >= 32) {
      return ((e >> 5) % (MR / 16)) * 16 + (e & 15);
    } else {
      return e >> 2;
    }
  }
  __device__ __forceinline__ static int piece_k4(int e) {  // which 4 k of the stage
    if constexpr (MR >= 32) {
      return ((e >> 5) / (MR / 16)) * 2 + ((e >> 4) & 1);
    } else {
      return e & 3;
    }
  }
  __device__ __forceinline__ XStager(const GemmParams& P, int64_t row0, int64_t kbeg, int64_t kend) {
#pragma unroll
    for (int u = 0; u < PIECES; ++u) {
      const int e = threadIdx.x + THREADS * u;
      const int64_t row = row0 + piece_row(e);
      const bool ok = e < NP && row < P.rows;
      kp[u] = ok ? kbeg + 4 * piece_k4(e) : kend;
      src[u] = ok ? P.x + row * P.kred + kbeg + 4 * piece_k4(e) : P.x;
    }
  }
  // A stage whose pieces may be ragged or absent (the slice's last stage, rows past M).
  __device__ __forceinline__ void copy(const GemmParams& P, int32_t* xt, int64_t kend, int st) const {
#pragma unroll
    for (int u = 0; u < PIECES; ++u) {
      const int e = threadIdx.x + THREADS * u;
      if (e >= NP) continue;
      const int64_t left = kend - (kp[u] + (int64_t)st * KC);  // valid k of the piece, if positive
      const int32_t* s = src[u] + (int64_t)st * KC;
      if constexpr (XV) {
        const int n = left >= 4 ? 16 : (left > 0 ? 4 * (int)left : 0);
        const uint32_t d = (uint32_t)__cvta_generic_to_shared(xt + 4 * e);
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(n ? s : P.x), "r"(n));
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          cp_async4(xt + 4 * e + i, i < left ? (const void*)(s + i) : (const void*)P.x, i < left);
      }
    }
  }
  // A stage whose pieces are all whole (every row present, all 16 k inside the slice): no checks.
  __device__ __forceinline__ void copy_full(int32_t* xt, int st) const {
#pragma unroll
    for (int u = 0; u < PIECES; ++u) {
      const int e = threadIdx.x + THREADS * u;
      if (e >= NP) continue;
      const int32_t* s = src[u] + (int64_t)st * KC;
      if constexpr (XV) {
        const uint32_t d = (uint32_t)__cvta_generic_to_shared(xt + 4 * e);
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(s));
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) cp_async4(xt + 4 * e + i, s + i, true);
      }
    }
  }
  __device__ __forceinline__ void transpose(const int32_t* xt, int32_t* xs) const {
    constexpr int XR = ClSmem<TMR>::XR;
#pragma unroll
    for (int u = 0; u < PIECES; ++u) {
      const int e = threadIdx.x + THREADS * u;
      if (e >= NP) continue;
      const int4 v = *reinterpret_cast<const int4*>(xt + 4 * e);
      int32_t* d = xs + (4 * piece_k4(e)) * XR + piece_row(e);
      d[0] = v.x;
      d[XR] = v.y;
      d[2 * XR] = v.z;
      d[3 * XR] = v.w;
    }
  }
};

// Blob path: the stage starting at k0 (a multiple of 16) is half (k0 / 16) % 2
// of packed chunk k0 / 32.  Thread t decodes 8 indices of column t % 64
// (indices past k_red decode to s = 0: the blob's padding is zero).
__device__ __forceinline__ void decode_codes(const GemmParams& P, int32_t* cs, int64_t col0, int64_t k0) {
  const int t = threadIdx.x;
  const int n = t & 63;
  const int h = t >> 6;                    // which 8 of the stage's 16 indices
  const int kk0 = (int)(k0 & 31) + 8 * h;  // first index within the 32-index chunk
  const int64_t col = col0 + n;
  uint32_t nib = 0u;
  uint2 bits = make_uint2(0u, 0u);
  if (col < P.cols) {
    const int64_t rec = (k0 / 32) * P.cols + col;
    nib = __ldg(reinterpret_cast<const uint32_t*>(P.blob + P.off_nib + rec * 16) + (kk0 >> 3));
    bits = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
  }
  int32_t* base = cs + (n >> 5) * 64 + (n & 31);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int k = 8 * h + i;  // index within the stage
    const int kk = kk0 + i;
    base[k * CW] = (int)((nib >> (4 * i)) & 15u);
    base[k * CW + 32] = (int)((bits.y >> kk) & 1u) - 2 * (int)((bits.x >> kk) & 1u);
  }
}

// Tile row of this thread's i-th row.
template <int TMR>
__device__ __forceinline__ int thread_row(int tm, int i) {
  if constexpr (TMR == 1) {
    return tm;
  } else {
    return (i >> 2) * 32 + 4 * tm + (i & 3);
  }
}

// The hot loop over one stage for this thread's rows I0 .. I0 + NI - 1 (whole
// row quads unless TMR = 1).
template <int TMR, int I0, int NI, typename Acc>
__device__ __forceinline__ void compute_stage(const int32_t* xs, const int32_t* cs, int tm, int tn,
                                              Acc (&acc)[NI][TN]) {
  constexpr int XR = ClSmem<TMR>::XR;
  const int32_t* cb = cs + ((tn * TN) >> 5) * 64 + ((tn * TN) & 31);
  const int32_t* xb = xs + (TMR == 1 ? tm : 4 * tm);
#pragma unroll
  for (int k = 0; k < KC; ++k) {
    int x[NI];
    if constexpr (TMR % 4 == 0) {
      static_assert(NI % 4 == 0 && I0 % 4 == 0, "whole row quads");
#pragma unroll
      for (int v = 0; v < NI / 4; ++v) {
        const int4 a = *reinterpret_cast<const int4*>(xb + k * XR + 32 * (I0 / 4 + v));
        x[4 * v] = a.x;
        x[4 * v + 1] = a.y;
        x[4 * v + 2] = a.z;
        x[4 * v + 3] = a.w;
      }
    } else {
      static_assert(TMR == 1 && NI == 1 && I0 == 0, "row mapping");
      x[0] = xb[k * XR];
    }
    const int4 s4 = *reinterpret_cast<const int4*>(cb + k * CW);
    const int4 g4 = *reinterpret_cast<const int4*>(cb + k * CW + 32);
    const int sh[TN] = {s4.x, s4.y, s4.z, s4.w};
    const int sg[TN] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
    for (int i = 0; i < NI; ++i) {
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const int t = x[i] >> sh[j];  // Eq. 1
        if constexpr (sizeof(Acc) == 4) {
          acc[i][j] += (uint32_t)sg[j] * (uint32_t)t;  // Eq. 2 + accumulate (mod 2^32)
        } else {
          acc[i][j] += (int64_t)sg[j] * (int64_t)t;
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

// One pass over the CTA's slice for this thread's rows I0 .. I0 + NI - 1 (the
// 32-bit path: all TMR rows at once; the 64-bit path of TMR = 8: two passes
// of one row quad each, so that its 64-bit accumulators fit the registers),
// then the cluster reduction of the tile rows those thread rows cover.
template <int TMR, bool XV, typename Acc, int I0, int NI>
__device__ __forceinline__ void run_cluster_tile(const GemmParams& P, ClSmem<TMR>& sm, cg::cluster_group& cl,
                                                 int64_t row0, int64_t col0, int64_t kbeg, int64_t kend,
                                                 uint32_t& amax_local) {
  constexpr int MR = 8 * TMR;
  const int t = threadIdx.x;
  const int tm = t % 8, tn = t / 8;
  const bool expanded = P.xcodes != nullptr;
  Acc acc[NI][TN];
#pragma unroll
  for (int i = 0; i < NI; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  // a trailing CTA of the cluster may have an empty slice: it stages nothing
  // and contributes zero partial sums
  const int nst = kend > kbeg ? (int)((kend - kbeg + KC - 1) / KC) : 0;
  const XStager<TMR, XV> xst(P, row0, kbeg, kend);
  const ExpandedCodeStager cst(P.xcodes, P.cols, P.kred, col0, kbeg);
  // stages whose x pieces and codes are all whole take the unchecked copies
  const bool whole_rows = row0 + MR <= P.rows && cst.b1;
  if (nst > 0) {
    xst.copy(P, sm.st.xt, kend, 0);
    if (expanded) cst.stage(P.xcodes, P.kred, sm.st.cs[0], 0);
    cp_async_commit();
    if (!expanded) decode_codes(P, sm.st.cs[0], col0, kbeg);
    cp_async_wait_all();
    xst.transpose(sm.st.xt, sm.st.xs[0]);
  }
  for (int st = 0; st < nst; ++st) {
    const int b = st & 1;
    const bool more = st + 1 < nst;
    const int64_t k1 = kbeg + (int64_t)(st + 1) * KC;
    __syncthreads();
    if (more) {
      if (whole_rows && k1 + KC <= kend) {
        xst.copy_full(sm.st.xt, st + 1);
        if (expanded) cst.stage_full(sm.st.cs[b ^ 1], st + 1);
      } else {
        xst.copy(P, sm.st.xt, kend, st + 1);
        if (expanded) cst.stage(P.xcodes, P.kred, sm.st.cs[b ^ 1], st + 1);
      }
      cp_async_commit();
    }
    compute_stage<TMR, I0, NI, Acc>(sm.st.xs[b], sm.st.cs[b], tm, tn, acc);
    if (more) {
      if (!expanded) decode_codes(P, sm.st.cs[b ^ 1], col0, k1);
      cp_async_wait_all();
      xst.transpose(sm.st.xt, sm.st.xs[b ^ 1]);
    }
  }
  __syncthreads();  // every thread is done with the staging buffers: they hold the partials next

  // this CTA's partial sums, [MR][64] row-major, 16 bytes per (row, 4 columns) for 32-bit
  Acc* red = reinterpret_cast<Acc*>(sm.red);
#pragma unroll
  for (int i = 0; i < NI; ++i) {
    Acc* dst = red + thread_row<TMR>(tm, I0 + i) * NT + tn * TN;
#pragma unroll
    for (int j = 0; j < TN; ++j) dst[j] = acc[i][j];
  }
  cl.sync();  // all partials of the cluster are written and visible

  const int rank = (int)cl.block_rank();
  const int cs_n = (int)cl.num_blocks();
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool vec_out = (P.cols % 4) == 0;
  // tile rows of this pass: all MR rows, or the 32 rows of one row quad
  constexpr int ROWS = TMR == 1 ? MR : 8 * NI;
  constexpr int ROW0 = TMR == 1 ? 0 : (I0 / 4) * 32;
  constexpr int GROUPS = ROWS * (NT / TN);  // (row, 4 columns) groups of the pass
  for (int gi = rank * THREADS + t; gi < GROUPS; gi += cs_n * THREADS) {
    const int r = ROW0 + gi / (NT / TN), c4 = gi % (NT / TN);
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

template <int TMR, bool XV>
__global__ void __launch_bounds__(THREADS, kMinBlocks) linear_cluster_kernel(const GemmParams P, int64_t k_per_cta) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  ClSmem<TMR>& sm = *reinterpret_cast<ClSmem<TMR>*>(smem_raw);
  cg::cluster_group cl = cg::this_cluster();
  const int64_t row0 = (int64_t)blockIdx.x * (8 * TMR);
  const int64_t col0 = (int64_t)blockIdx.y * NT;
  const int64_t kbeg = (int64_t)cl.block_rank() * k_per_cta;
  const int64_t kend = min(P.kred, kbeg + k_per_cta);
  uint32_t amax_local = 0;
  if (tile_int32_exact(P, col0)) {
    run_cluster_tile<TMR, XV, uint32_t, 0, TMR>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
  } else if constexpr (TMR == 8) {
    run_cluster_tile<TMR, XV, int64_t, 0, 4>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
    run_cluster_tile<TMR, XV, int64_t, 4, 4>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
  } else {
    run_cluster_tile<TMR, XV, int64_t, 0, TMR>(P, sm, cl, row0, col0, kbeg, kend, amax_local);
  }
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

// How many clusters of cs CTAs the device can hold at once (0: not
// launchable), queried once per process and size.
template <int TMR, bool XV>
int active_clusters(int cs) {
  static int cache[kMaxCluster + 1] = {0};
  static bool attrs_set = false;
  static std::mutex mu;  // the cache is shared by every host thread
  std::lock_guard<std::mutex> lock(mu);
  if (cs < 1 || cs > kMaxCluster) return 0;
  if (cache[cs] != 0) return cache[cs] > 0 ? cache[cs] : 0;
  auto kern = linear_cluster_kernel<TMR, XV>;
  if (!attrs_set) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(ClSmem<TMR>)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
      (void)cudaGetLastError();
      return 0;
    }
    attrs_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, 1, cs);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = sizeof(ClSmem<TMR>);
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 1;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = cs;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();  // a refused size
    n = 0;
  }
  cache[cs] = n > 0 ? n : -1;
  return n;
}

template <int TMR, bool XV>
cudaError_t launch_tmr(const GemmParams& p, cudaStream_t st) {
  constexpr int MR = 8 * TMR;
  const int64_t tiles = ((p.rows + MR - 1) / MR) * ((p.cols + NT - 1) / NT);
  const int64_t stages = (p.kred + KC - 1) / KC;
  // the cluster size: at most one wave of CTAs and at least one stage per
  // CTA, chosen for the least time counted as waves x stages per CTA, where
  // a wave is the number of clusters the device holds at once (trailing
  // slices may still be empty)
  const int64_t cs_max = std::max<int64_t>(
      std::min<int64_t>(std::min<int64_t>(slots() / std::max<int64_t>(tiles, 1), kMaxCluster), stages), 1);
  int64_t cs = 0, best = 0;
  for (int64_t c = 1; c <= cs_max; ++c) {
    const int n = active_clusters<TMR, XV>((int)c);
    if (n <= 0) continue;
    const int64_t cost = ((tiles + n - 1) / n) * ((stages + c - 1) / c);
    if (cs == 0 || cost < best) {
      best = cost;
      cs = c;
    }
  }
  if (cs == 0) return cudaErrorLaunchOutOfResources;
  const int64_t stages_per_cta = (stages + cs - 1) / cs;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((p.rows + MR - 1) / MR), (unsigned)((p.cols + NT - 1) / NT), (unsigned)cs);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = sizeof(ClSmem<TMR>);
  cfg.stream = st;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 1;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = (unsigned)cs;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, linear_cluster_kernel<TMR, XV>, p, stages_per_cta * KC);
}

template <bool XV>
cudaError_t launch_xv(const GemmParams& p, cudaStream_t st) {
  if (p.rows <= 8) return launch_tmr<1, XV>(p, st);
  if (p.rows <= 32) return launch_tmr<4, XV>(p, st);
  return launch_tmr<8, XV>(p, st);
}

}  // namespace

bool linear_cluster_preferred(const GemmParams& p) {
  // the 128 x 64 tiles of shift_gemm.cu would not fill the SMs three times over
  const int64_t gemm_ctas = ((p.rows + 127) / 128) * ((p.cols + NT - 1) / NT);
  return gemm_ctas < 3 * (int64_t)sm_count() && (p.cols + NT - 1) / NT <= 65535 && (p.rows + 7) / 8 <= (int64_t)INT32_MAX;
}

cudaError_t launch_linear_cluster(const GemmParams& p, cudaStream_t st) {
  // 16-byte x pieces need 16-byte aligned rows: K a multiple of 4 (x itself is 16-byte aligned)
  const bool xv = (p.kred % 4) == 0 && (reinterpret_cast<uintptr_t>(p.x) & 15) == 0;
  return xv ? launch_xv<true>(p, st) : launch_xv<false>(p, st);
}

}  // namespace ds
