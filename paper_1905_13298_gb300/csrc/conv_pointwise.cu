// Pointwise (1x1) ConvShift as a shift GEMM over pixels (DeepShift Eq. 1-3).
//
//   y[n][k][oh][ow] = sat32( b[k] + sum_c s[k][c] * (x[n][c][oh*sig][ow*sig] >> -p[k][c]) )
//
// A 1x1 convolution has no window to reuse, so it runs as a GEMM whose rows
// are output pixels (all images), columns are output channels and whose
// reduction runs over input channels.  The activation tile of a stage is
// staged channel-major ([16 channels][128 pixels]): for stride 1 every
// 16-byte chunk of 4 pixels is one cp.async, for stride 2 four 4-byte copies.
// A thread owns 8 pixels (two quads 64 apart, so a warp's 16-byte loads are
// contiguous) and 8 channels; per term the hot loop is one SHF and one IMAD.
// 128 threads at 128 registers and 32 KB of shared memory: 4 CTAs per SM.
// Codes come from the expanded execution layout (cp.async) or are decoded
// from the packed blob per stage (ExpandedCodeStager: each thread's code
// pieces and source address are fixed, advancing by 16 channels per stage).
// The epilogue writes each (quad, channel)
// as one 16-byte store when OH*OW is a multiple of 4.  Accumulator width as
// in shift_gemm.cu.
//
// Split reduction (layers whose grid would not fill the SMs, e.g. 2048
// input channels on 7x7 maps, or a 1x1/2 downsample at batch 32): grid.z
// CTAs share a tile's stages.  Normally the CTAs form a thread-block
// cluster, and each rank reduces a share of the tile's partial sums over all
// ranks through distributed shared memory and applies the epilogue itself.
// With a workspace (the chained forward) a grid below a sixteenth of the SM
// slots instead adds its exact partial sums into the workspace with 64-bit
// atomics, and the finalize kernel of conv_direct.cu applies the epilogue.
#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>

#include "ds_common.cuh"

namespace cg = cooperative_groups;

namespace ds {
namespace {

constexpr int MT = 128;       // pixels per CTA
constexpr int NT = 64;        // channels per CTA
constexpr int TN = 8;         // channels per thread
constexpr int PG = MT / 8;    // pixel groups (two quads each)
constexpr int THREADS = 128;  // PG x (NT / TN)
constexpr int KC = 16;        // input channels per stage (half of a packed 32-index chunk)
constexpr int NB = NT / 32;   // 32-channel blocks of the expanded layout per CTA
constexpr int QUADS = MT / 4;
constexpr int kMaxCluster = 16;  // CTAs per thread-block cluster (non-portable maximum)
constexpr int kChainPwClusterMaxTarget = 16;  // see pw_stages_per_split
// resident CTAs of the device (4 per SM)
inline int64_t slots() { return (int64_t)sm_count() * 4; }
static_assert(PG * (NT / TN) == THREADS && THREADS % QUADS == 0, "tile shape");

struct __align__(16) PwSmem {
  int32_t xs[2][KC * MT];
  int32_t cs[2][KC * 2 * NT];  // per input channel: NB blocks of {32 shifts, 32 signs}
};

// This thread's staging assignment: pixel quad q = t % 32 of the tile, input
// channels t / 32 + 4 j.  Input offsets of the quad's 4 pixels (channel 0).
struct QuadCtx {
  int64_t off[4];
  bool valid[4];
  bool vec;  // the 4 pixels are consecutive and 16-byte aligned in memory
};

template <bool STRIDED>
__device__ __forceinline__ QuadCtx quad_ctx(const GemmParams& P, int64_t m0) {
  QuadCtx q;
  const int64_t OHW = (int64_t)P.OH * P.OW;
  const int64_t CHW = (int64_t)P.C * P.H * P.W;
  const int64_t mq = m0 + 4 * (threadIdx.x % QUADS);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t m = mq + i;
    q.valid[i] = m < P.rows;
    const int64_t n = q.valid[i] ? m / OHW : 0;
    const int64_t pix = q.valid[i] ? m - n * OHW : 0;
    if constexpr (STRIDED) {
      const int oh = (int)(pix / P.OW), ow = (int)(pix - (pix / P.OW) * P.OW);
      q.off[i] = n * CHW + (int64_t)oh * P.sh * P.W + (int64_t)ow * P.sw;
    } else {
      q.off[i] = n * CHW + pix;
    }
  }
  // 16-byte copies need every channel's quad aligned: offset and channel stride multiples of 4 words
  q.vec = !STRIDED && q.valid[3] && (q.off[3] == q.off[0] + 3) && ((q.off[0] & 3) == 0) &&
          ((((int64_t)P.H * P.W) & 3) == 0) && ((reinterpret_cast<uintptr_t>(P.x) & 15) == 0);
  return q;
}

template <bool STRIDED>
__device__ __forceinline__ void stage_x(const GemmParams& P, int32_t* xs, const QuadCtx& q, int c0) {
  const int64_t HW = (int64_t)P.H * P.W;
  const int qi = threadIdx.x % QUADS;
  constexpr int ROWS = THREADS / QUADS;  // channel rows per pass
  const int cl0 = (int)(threadIdx.x / QUADS);
  const int32_t* xc = P.x + (int64_t)(c0 + cl0) * HW;  // this thread's first channel of the stage
#pragma unroll
  for (int j = 0; j < KC / ROWS; ++j) {
    const int cl = cl0 + ROWS * j;
    const int32_t* xj = xc + (int64_t)(ROWS * j) * HW;
    int32_t* dst = xs + cl * MT + 4 * qi;
    const bool cok = c0 + cl < P.C;
    if (!STRIDED && q.vec) {
      cp_async16(dst, cok ? (const void*)(xj + q.off[0]) : (const void*)P.x, cok);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool ok = cok && q.valid[i];
        cp_async4(dst + i, ok ? (const void*)(xj + q.off[i]) : (const void*)P.x, ok);
      }
    }
  }
}

// Blob path: stage st covers reduction indices [16 st, 16 st + 16), half
// st % 2 of packed chunk st / 2.  Thread t decodes 8 indices of column t % 64
// (indices past k_red decode to s = 0: the blob's padding is zero).
__device__ __forceinline__ void decode_codes(const GemmParams& P, int32_t* cs, int64_t col0, int st) {
  const int t = threadIdx.x;
  const int n = t & 63;
  const int h = t >> 6;                   // which 8 of the stage's 16 indices
  const int kk0 = 16 * (st & 1) + 8 * h;  // first index within the 32-index chunk
  const int64_t col = col0 + n;
  uint32_t nib = 0u;
  uint2 bits = make_uint2(0u, 0u);
  if (col < P.cols) {
    const int64_t rec = (int64_t)(st >> 1) * P.cols + col;
    nib = __ldg(reinterpret_cast<const uint32_t*>(P.blob + P.off_nib + rec * 16) + (kk0 >> 3));
    bits = __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
  }
  int32_t* base = cs + (n >> 5) * 64 + (n & 31);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int k = 8 * h + i;  // index within the stage
    const int kk = kk0 + i;
    base[k * 2 * NT] = (int)((nib >> (4 * i)) & 15u);
    base[k * 2 * NT + 32] = (int)((bits.y >> kk) & 1u) - 2 * (int)((bits.x >> kk) & 1u);
  }
}

template <int I0, int NI, typename Acc>
__device__ __forceinline__ void compute_stage(const int32_t* xs, const int32_t* cs, int tm, int tn,
                                              Acc (&acc)[NI][TN]) {
  const int32_t* cbase = cs + ((tn * TN) >> 5) * 64 + ((tn * TN) & 31);
#pragma unroll 2
  for (int k = 0; k < KC; ++k) {
    int x[8];
    {
      const int4 a = *reinterpret_cast<const int4*>(xs + k * MT + 4 * tm);
      const int4 b = *reinterpret_cast<const int4*>(xs + k * MT + MT / 2 + 4 * tm);
      x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
      x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    }
    int sh[TN], sg[TN];
#pragma unroll
    for (int v = 0; v < TN / 4; ++v) {
      const int4 s0 = *reinterpret_cast<const int4*>(cbase + k * 2 * NT + 4 * v);
      const int4 g0 = *reinterpret_cast<const int4*>(cbase + k * 2 * NT + 32 + 4 * v);
      sh[4 * v] = s0.x; sh[4 * v + 1] = s0.y; sh[4 * v + 2] = s0.z; sh[4 * v + 3] = s0.w;
      sg[4 * v] = g0.x; sg[4 * v + 1] = g0.y; sg[4 * v + 2] = g0.z; sg[4 * v + 3] = g0.w;
    }
    // channel-outer order: consecutive SHF / IMAD share their shift / sign operand
#pragma unroll
    for (int j = 0; j < TN; ++j) {
#pragma unroll
      for (int i = 0; i < NI; ++i) {
        const int xv = x[I0 + i];
        const int t = xv >> sh[j];  // Eq. 1
        if constexpr (sizeof(Acc) == 4) {
          acc[i][j] += (uint32_t)sg[j] * (uint32_t)t;  // Eq. 2 + accumulate (mod 2^32)
        } else {
          acc[i][j] += (int64_t)sg[j] * (int64_t)t;
        }
      }
    }
  }
}

// Output value of an exact (64-bit) or proven-exact (32-bit) sum plus bias:
// saturated to int32 (the 64-bit path; the 32-bit path cannot leave it).
template <typename Acc>
__device__ __forceinline__ int32_t finish_sum(Acc a, int32_t b) {
  if constexpr (sizeof(Acc) == 4) {
    return (int32_t)(a + (uint32_t)b);
  } else {
    int64_t v = a + (int64_t)b;
    v = v > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : v;
    v = v < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : v;
    return (int32_t)v;
  }
}

// Cluster split: this CTA's partial sums go to its shared memory as
// red[(thread * NI + i) * TN + j]; every rank has the same tile mapping, so
// entry f of every rank belongs to the same output (pixel slot i of thread
// f / NI, its channels j).  Rank r sums the entries f = r * THREADS + t
// (mod cs * THREADS) over all ranks through distributed shared memory (the
// 32-bit partials are exact whenever the bound holds: each is a subset of the
// terms) and applies the epilogue.  The second cluster barrier keeps every
// rank's shared memory alive until the remote reads end.
template <int I0, int NI, typename Acc>
__device__ __forceinline__ void cluster_epilogue(const GemmParams& P, PwSmem& sm, int64_t m0, int64_t col0,
                                                 const Acc (&acc)[NI][TN], uint32_t& amax_local) {
  static_assert(THREADS * NI * TN * sizeof(Acc) <= sizeof(PwSmem), "partials fit the staging buffers");
  const int t = threadIdx.x;
  Acc* red = reinterpret_cast<Acc*>(&sm);
#pragma unroll
  for (int i = 0; i < NI; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) red[(t * NI + i) * TN + j] = acc[i][j];
  cg::cluster_group cl = cg::this_cluster();
  cl.sync();  // all partials written
  const int rank = (int)cl.block_rank();
  const int cs = (int)cl.num_blocks();
  const int64_t OHW = (int64_t)P.OH * P.OW;
  const bool relu = (P.flags & DS_RELU) != 0;
  const int32_t* resid = (P.flags & DS_RESIDUAL) ? P.residual : nullptr;
  for (int f = rank * THREADS + t; f < THREADS * NI; f += cs * THREADS) {
    const int ft = f / NI, i = f - ft * NI;
    const int li = I0 + i;
    const int64_t m = m0 + 4 * (ft % PG) + (li & 3) + (MT / 2) * (li >> 2);
    Acc sum[TN];
#pragma unroll
    for (int j = 0; j < TN; ++j) sum[j] = 0;
    for (int q = 0; q < cs; ++q) {
      const Acc* src = cl.map_shared_rank(red, q) + f * TN;
      if constexpr (sizeof(Acc) == 4) {
#pragma unroll
        for (int v = 0; v < TN / 4; ++v) {
          const uint4 w = *reinterpret_cast<const uint4*>(src + 4 * v);
          sum[4 * v] += w.x;
          sum[4 * v + 1] += w.y;
          sum[4 * v + 2] += w.z;
          sum[4 * v + 3] += w.w;
        }
      } else {
#pragma unroll
        for (int v = 0; v < TN / 2; ++v) {
          const longlong2 w = *reinterpret_cast<const longlong2*>(src + 2 * v);
          sum[2 * v] += w.x;
          sum[2 * v + 1] += w.y;
        }
      }
    }
    if (m >= P.rows) continue;
    const int64_t n = m / OHW;
    const int64_t base = n * P.cols * OHW + (m - n * OHW);
    const int64_t c0 = col0 + (ft / PG) * TN;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int64_t col = c0 + j;
      if (col >= P.cols) break;
      const int64_t idx = base + col * OHW;
      int32_t o = finish_sum<Acc>(sum[j], P.bias != nullptr ? __ldg(P.bias + col) : 0);
      if (resid != nullptr) o = add_sat(o, __ldg(resid + idx));
      if (relu) o = max(o, 0);
      amax_local = max(amax_local, uabs(o));
      P.y[idx] = o;
    }
  }
  cl.sync();  // no rank reuses its shared memory (next pass) or exits while another reads it
}

template <bool STRIDED, bool CL, int I0, int NI, typename Acc>
__device__ __forceinline__ void run_tile(const GemmParams& P, PwSmem& sm, int64_t m0, int64_t col0,
                                         const QuadCtx& q, int st_begin, int st_end, uint32_t& amax_local) {
  const int t = threadIdx.x;
  const int tm = t % PG, tn = t / PG;
  const bool expanded = P.xcodes != nullptr;
  Acc acc[NI][TN];
#pragma unroll
  for (int i = 0; i < NI; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  static_assert(KC == 16 && NB == 2 && THREADS == 128, "ExpandedCodeStager's stage shape");
  const ExpandedCodeStager cst(P.xcodes, P.cols, P.kred, col0, (int64_t)st_begin * KC);
  if (!CL || st_begin < st_end) {  // a trailing rank of a cluster may have no stage: zero partial sums
    stage_x<STRIDED>(P, sm.xs[0], q, st_begin * KC);
    if (expanded) cst.stage(P.xcodes, P.kred, sm.cs[0], 0);
    cp_async_commit();
    if (!expanded) decode_codes(P, sm.cs[0], col0, st_begin);
    cp_async_wait_all();
  }
  for (int st = st_begin; st < st_end; ++st) {
    const int b = (st - st_begin) & 1;
    const bool more = st + 1 < st_end;
    __syncthreads();
    if (more) {
      stage_x<STRIDED>(P, sm.xs[b ^ 1], q, (st + 1) * KC);
      if (expanded) cst.stage(P.xcodes, P.kred, sm.cs[b ^ 1], st + 1 - st_begin);
      cp_async_commit();
    }
    compute_stage<I0, NI, Acc>(sm.xs[b], sm.cs[b], tm, tn, acc);
    if (more) {
      if (!expanded) decode_codes(P, sm.cs[b ^ 1], col0, st + 1);
      cp_async_wait_all();
    }
  }
  __syncthreads();  // a second pass (64-bit path) or the cluster partials reuse the buffers

  if constexpr (CL) {
    cluster_epilogue<I0, NI, Acc>(P, sm, m0, col0, acc, amax_local);
    return;
  }
  const int64_t OHW = (int64_t)P.OH * P.OW;
  if (P.split_acc != nullptr) {
    // split reduction: exact partial sums (a subset of the terms, so 32-bit
    // partials are exact whenever the full sum is) into the int64 workspace
#pragma unroll
    for (int i = 0; i < NI; ++i) {
      const int li = I0 + i;
      const int64_t m = m0 + 4 * tm + (li & 3) + (MT / 2) * (li >> 2);
      if (m >= P.rows) continue;
      const int64_t n = m / OHW;
      const int64_t base = n * P.cols * OHW + (m - n * OHW);
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const int64_t col = col0 + tn * TN + j;
        if (col >= P.cols) break;
        const int64_t v = sizeof(Acc) == 4 ? (int64_t)(int32_t)acc[i][j] : (int64_t)acc[i][j];
        atomicAdd(reinterpret_cast<unsigned long long*>(P.split_acc + base + col * OHW), (unsigned long long)v);
      }
    }
    return;
  }

  // fused epilogue: bias, saturation (64-bit path), residual, ReLU, amax.
  // The thread's pixels are two quads of 4 consecutive output pixels.  When
  // OH*OW is a multiple of 4 a quad lies inside one image and starts on a
  // 16-byte boundary, so each (quad, channel) is one 16-byte load / store.
  const bool relu = (P.flags & DS_RELU) != 0;
  const int32_t* resid = (P.flags & DS_RESIDUAL) ? P.residual : nullptr;
  const bool vec = ((OHW & 3) == 0) && (resid == nullptr || (reinterpret_cast<uintptr_t>(resid) & 15) == 0);
  int32_t bcol[TN];
#pragma unroll
  for (int j = 0; j < TN; ++j) {
    const int64_t col = col0 + tn * TN + j;
    bcol[j] = (P.bias != nullptr && col < P.cols) ? __ldg(P.bias + col) : 0;
  }
  auto finish = [](Acc a, int32_t b) -> int32_t {
    if constexpr (sizeof(Acc) == 4) {
      return (int32_t)(a + (uint32_t)b);
    } else {
      int64_t v = a + (int64_t)b;
      v = v > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : v;
      v = v < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : v;
      return (int32_t)v;
    }
  };
  if (vec) {
#pragma unroll
    for (int qd = 0; qd < NI / 4; ++qd) {
      const int64_t mq = m0 + 4 * tm + (MT / 2) * ((I0 >> 2) + qd);
      if (mq >= P.rows) continue;  // rows = N * OH * OW is a multiple of 4: quads are whole
      const int64_t n = mq / OHW;  // once per quad
      const int64_t base = n * P.cols * OHW + (mq - n * OHW);
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const int64_t col = col0 + tn * TN + j;
        if (col >= P.cols) break;
        const int64_t idx = base + col * OHW;
        int32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) o[e] = finish(acc[4 * qd + e][j], bcol[j]);
        if (resid != nullptr) {
          const int4 r = __ldg(reinterpret_cast<const int4*>(resid + idx));
          o[0] = add_sat(o[0], r.x);
          o[1] = add_sat(o[1], r.y);
          o[2] = add_sat(o[2], r.z);
          o[3] = add_sat(o[3], r.w);
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (relu) o[e] = max(o[e], 0);
          amax_local = max(amax_local, uabs(o[e]));
        }
        *reinterpret_cast<int4*>(P.y + idx) = make_int4(o[0], o[1], o[2], o[3]);
      }
    }
    return;
  }
#pragma unroll
  for (int i = 0; i < NI; ++i) {
    const int li = I0 + i;
    const int64_t m = m0 + 4 * tm + (li & 3) + (MT / 2) * (li >> 2);
    if (m >= P.rows) continue;
    const int64_t n = m / OHW;  // once per pixel
    const int64_t base = n * P.cols * OHW + (m - n * OHW);
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int64_t col = col0 + tn * TN + j;
      if (col >= P.cols) break;
      const int64_t idx = base + col * OHW;
      int32_t o = finish(acc[i][j], bcol[j]);
      if (resid != nullptr) o = add_sat(o, __ldg(resid + idx));
      if (relu) o = max(o, 0);
      amax_local = max(amax_local, uabs(o));
      P.y[idx] = o;
    }
  }
}

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

// The cluster variant allows 3 CTAs per SM (168 registers): at 4 its reduction
// epilogue spilled into the hot loop, and it runs only on grids that do not
// fill the SMs anyway.
template <bool STRIDED, bool CL>
__global__ void __launch_bounds__(THREADS, CL ? 3 : 4) conv_pointwise_kernel(const GemmParams P, int stages_per_split) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  PwSmem& sm = *reinterpret_cast<PwSmem*>(smem_raw);
  const int64_t m0 = (int64_t)blockIdx.x * MT;
  const int64_t col0 = (int64_t)blockIdx.y * NT;
  const int n_stages = (P.C + KC - 1) / KC;
  const int st_begin = blockIdx.z * stages_per_split;
  const int st_end = min(n_stages, st_begin + stages_per_split);
  const QuadCtx q = quad_ctx<STRIDED>(P, m0);
  uint32_t amax_local = 0;
  if (tile_int32_exact(P, col0)) {
    run_tile<STRIDED, CL, 0, 8, uint32_t>(P, sm, m0, col0, q, st_begin, st_end, amax_local);
  } else {
    run_tile<STRIDED, CL, 0, 4, int64_t>(P, sm, m0, col0, q, st_begin, st_end, amax_local);
    run_tile<STRIDED, CL, 4, 4, int64_t>(P, sm, m0, col0, q, st_begin, st_end, amax_local);
  }
  if (P.amax_out != nullptr && P.split_acc == nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

// Stages per CTA of an atomic split reduction (n_stages: none).  Only with a
// workspace that holds the int64 partial sums, and only for a grid below a
// sixteenth of the SM slots: a larger under-filled grid splits over a
// cluster, as without a workspace (measured: the atomics, the memset and the
// finalize cost more than the cluster barriers; ResNet18 batch 32 4.75 ->
// 4.68 ms per forward, batch 8 1.60 -> 1.58 ms); then it targets two waves.
int pw_stages_per_split(const GemmParams& p, size_t split_capacity) {
  const int n_stages = (p.C + KC - 1) / KC;
  const int64_t ctas = ((p.rows + MT - 1) / MT) * ((p.cols + NT - 1) / NT);
  const size_t need = (size_t)p.rows * p.cols * sizeof(int64_t);
  if (split_capacity < need || ctas >= slots() || n_stages < 2) return n_stages;
  if (slots() / std::max<int64_t>(ctas, 1) <= kChainPwClusterMaxTarget) return n_stages;
  const int want = (int)std::min<int64_t>(n_stages, (2 * slots() + ctas - 1) / ctas);
  return (n_stages + want - 1) / want;
}

template <bool STRIDED, bool CL>
bool set_pw_attributes() {
  // once per process, thread-safe (see conv_direct.cu)
  static const bool ok = [] {
    const bool r = cudaFuncSetAttribute(conv_pointwise_kernel<STRIDED, CL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)sizeof(PwSmem)) == cudaSuccess &&
                   (!CL || cudaFuncSetAttribute(conv_pointwise_kernel<STRIDED, CL>,
                                                cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess);
    if (!r) (void)cudaGetLastError();
    return r;
  }();
  return ok;
}

// How many clusters of cs CTAs the device holds at once (0: none); queried
// once per process and size.
template <bool STRIDED>
int pw_max_clusters(int cs) {
  if (cs < 2 || cs > kMaxCluster || !set_pw_attributes<STRIDED, true>()) return 0;
  static int cache[kMaxCluster + 1] = {0};
  static std::mutex mu;  // shared by every host thread
  std::lock_guard<std::mutex> lock(mu);
  if (cache[cs] != 0) return cache[cs] > 0 ? cache[cs] : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, 1, cs);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = sizeof(PwSmem);
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 1;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = cs;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, conv_pointwise_kernel<STRIDED, true>, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    n = 0;
  }
  cache[cs] = n > 0 ? n : -1;
  return n > 0 ? n : 0;
}

// Cluster size of a standalone call whose grid does not fill every SM slot
// once: the size with the least time, counted as waves x stages per rank
// (as the direct kernel chooses it); 1: no split.
template <bool STRIDED>
int pw_cluster_size(const GemmParams& p) {
  const int n_stages = (p.C + KC - 1) / KC;
  const int64_t tiles = ((p.rows + MT - 1) / MT) * ((p.cols + NT - 1) / NT);
  if (tiles >= slots() || n_stages < 2) return 1;
  int cs = 1;
  int64_t best = ((tiles + slots() - 1) / std::max<int64_t>(slots(), 1)) * n_stages;
  for (int c = 2; c <= std::min(kMaxCluster, n_stages); ++c) {
    const int n = pw_max_clusters<STRIDED>(c);
    if (n <= 0) continue;
    const int64_t cost = ((tiles + n - 1) / n) * ((n_stages + c - 1) / c);
    if (cost < best) {
      best = cost;
      cs = c;
    }
  }
  return cs;
}

template <bool STRIDED>
cudaError_t launch_pw(const GemmParams& p, cudaStream_t st) {
  const size_t smem = sizeof(PwSmem);
  if (!set_pw_attributes<STRIDED, false>()) return cudaErrorInvalidValue;
  const int n_stages = (p.C + KC - 1) / KC;
  const int sps = pw_stages_per_split(p, p.split_acc ? p.split_capacity : 0);
  const int splits = (n_stages + sps - 1) / sps;
  GemmParams q = p;
  const dim3 grid1((unsigned)((p.rows + MT - 1) / MT), (unsigned)((p.cols + NT - 1) / NT), 1u);
  if (splits == 1) {
    q.split_acc = nullptr;
    int cs = pw_cluster_size<STRIDED>(p);
    const int sps_cl = (n_stages + cs - 1) / cs;
    cs = (n_stages + sps_cl - 1) / sps_cl;  // every rank gets at least one stage
    if (cs >= 2) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(grid1.x, grid1.y, (unsigned)cs);
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
      return cudaLaunchKernelEx(&cfg, conv_pointwise_kernel<STRIDED, true>, q, sps_cl);
    }
  } else {
    cudaError_t e = prepare_split_scratch(q, st);
    if (e != cudaSuccess) return e;
  }
  const dim3 grid(grid1.x, grid1.y, (unsigned)splits);
  conv_pointwise_kernel<STRIDED, false><<<grid, THREADS, smem, st>>>(q, sps);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || splits == 1) return e;
  return launch_split_finalize(q, st);
}

}  // namespace

bool conv_pointwise_supported(const GemmParams& p) {
  return p.R == 1 && p.S == 1 && p.ph == 0 && p.pw == 0 && p.sh >= 1 && p.sw >= 1 && p.cols <= 65535LL * NT &&
         (p.rows + MT - 1) / MT <= (int64_t)INT32_MAX;
}

size_t conv_pointwise_split_bytes(const GemmParams& p) {
  if (!conv_pointwise_supported(p)) return 0;
  const int n_stages = (p.C + KC - 1) / KC;
  if (pw_stages_per_split(p, ~(size_t)0) >= n_stages) return 0;
  return (size_t)p.rows * p.cols * sizeof(int64_t);
}

cudaError_t launch_conv2d_pointwise(const GemmParams& p, cudaStream_t st) {
  const bool strided = p.sh != 1 || p.sw != 1;
  return strided ? launch_pw<true>(p, st) : launch_pw<false>(p, st);
}

}  // namespace ds
