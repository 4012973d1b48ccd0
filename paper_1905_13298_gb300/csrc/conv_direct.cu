// ConvShift forward, direct (halo-tile) kernel (DeepShift Eq. 1-3, Sec. 4).
//
//   y[n][k][oh][ow] = sat32( b[k] + sum_{c,r,s} s_w * (xpad[n][c][oh*sig + r][ow*sig + s] >> -p) )
//
// CTA tile: one image, TH output rows x GW groups of TM consecutive output
// columns, NT output channels (256 threads, 8 warps).  A thread owns one
// group (TM pixels of one row) and TN = 4 channels.  Per chunk of CC input
// channels (one pipeline stage) the CTA stages into shared memory
//   * the input window of every group, zero outside the image, as a "slot"
//     of WSP words (WS = (TM-1)*sig + S values, padded to 16 bytes and to a
//     stride of 4 mod 8 words), so that a thread reads the window of one
//     kernel row with ceil(WS/4) vector loads;
//   * the codes of the chunk's taps as 32-bit shift / sign words, one row of
//     NT channels per tap: copied with 16-byte cp.async from the expanded
//     execution layout when the layer has one, else decoded from the packed
//     blob (one item of at most 16 taps of one channel per thread).
// For each (c, r) a thread loads its window once and reuses it for the S
// taps of that row (sliding window); per term the hot loop issues one
// arithmetic right shift (ALU pipe) and one multiply-add by the sign (FMA
// pipe).  Stages are double buffered with one barrier per stage.
//
// Accumulator width as in shift_gemm.cu: 32-bit when the launch bound proves
// it exact for the CTA's channels, else a 64-bit pass per half of the pixels.
#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>

#include "ds_common.cuh"

namespace cg = cooperative_groups;

namespace ds {
namespace {

constexpr int TN = 4;                   // output channels per thread
constexpr int NT = 32;                  // output channels per CTA
constexpr int CG = NT / TN;             // channel groups per CTA
constexpr int kMaxThreads = 256;        // 8 warps: every SM sub-partition gets the same share
constexpr int kSmemBudget = 74 * 1024;  // 3 CTAs per SM
// resident CTAs of the device (3 per SM)
inline int64_t slots() { return (int64_t)sm_count() * 3; }
constexpr int kMaxCluster = 16;         // CTAs per thread-block cluster (non-portable maximum)
constexpr int kChainClusterMaxTarget = 2;  // see choose_geom

// The CTA tiles run over the stacked output rows gr = n * OH + oh of all
// images, so a tile may span image boundaries (small feature maps, batch 1).
// In "stacked input" coordinates image n's zero-padded rows are
// n * HP + ihp (HP = H + 2 * pad); output row (n, oh) reads stacked rows
// n * HP + oh * sig + r.  A tile's halo is the contiguous stacked range its
// rows read, HR rows at most.
struct DirectGeom {
  int TH, GW;        // output rows and pixel groups per row per CTA
  int threads;       // TH * GW * CG
  int CC;            // input channels per stage
  int HR, HP;        // halo rows per tile, padded input height
  int N;             // images
  int taps;          // CC * R * S
  int n_stages;      // ceil(C / CC)
  int halo_words;    // CC * HR * GW * WSP
  int code_words;    // taps * 2 * NT
  int run;           // taps per decode item (blob path)
  int tiles_w, tiles_h;
  int splits, stages_per_split;  // split reduction over the stages
  int cluster;                   // > 1: the splits form one thread-block cluster (reduction in DSMEM)
  int pairs;                     // stride 2: stage the halo with 8-byte copies (even W, odd padding)
  FastDiv dGW, dHR, dHP;         // dividers of the halo staging
};

template <int SIG, int S, int TM>
struct Win {
  static constexpr int WS = (TM - 1) * SIG + S;  // window values
  // Stride 2: the slot starts one column before the window (word D = 1 holds
  // its first value), so that with an odd padding and an even row length
  // (every ResNet stride-2 layer) the slot starts on an even column and is
  // staged with 8-byte copies.
  static constexpr int D = SIG == 2 ? 1 : 0;
  static constexpr int WV = (WS + D + 3) / 4;  // 16-byte loads per window
  // slot stride in words: 16-byte aligned and 4 mod 8, so that the 4-byte
  // copies of 32 consecutive slots fill 8 bank groups (4-way at most) rather
  // than 2 (16-way) when the window is a multiple of 8 words
  static constexpr int WSP = WV * 4 + (WV % 2 == 0 ? 4 : 0);
};

// Stage the group windows of input channels [c0, c0 + CC) for halo rows
// n0 * HP + off0 + [0, HR) (stacked coordinates): one slot (channel, halo row,
// group) per thread at a time; zero in padding rows, outside the image and
// for channels >= C.
template <int SIG, int S, int TM>
__device__ __forceinline__ void stage_halo(const GemmParams& P, const DirectGeom G, int32_t* halo, int n0,
                                           int off0, int iw0, int c0) {
  using WN = Win<SIG, S, TM>;
  const int64_t HW = (int64_t)P.H * P.W;
  const int nslots = G.CC * G.HR * G.GW;
  for (int sl = threadIdx.x; sl < nslots; sl += G.threads) {
    const int row = fdiv(sl, G.dGW);  // (channel, halo row)
    const int g = sl - row * G.GW;
    const int cl = fdiv(row, G.dHR);
    const int hr = row - cl * G.HR;
    const int c = c0 + cl;
    const int o = off0 + hr;  // stacked row, counted from image n0's first padded row
    const int di = fdiv(o, G.dHP);
    const int ni = n0 + di;
    const int ih = o - di * G.HP - P.ph;
    const int iws = iw0 + g * TM * SIG - WN::D;  // first staged column
    int32_t* dst = halo + sl * WN::WSP;
    const bool row_ok = (c < P.C) && (ni < G.N) && ((unsigned)ih < (unsigned)P.H);
    const int32_t* src = P.x + ((int64_t)ni * P.C + c) * HW + (int64_t)ih * P.W + iws;
    constexpr int NW = WN::WS + WN::D;  // words staged per slot
    // Every slot takes the same predicated copies (zero fill outside the
    // image): an unpredicated branch for interior slots made the warps that
    // also hold edge slots run both paths (measured: the uniform form is 2.8%
    // faster on the 56 x 56 3x3/1 layer).
    if constexpr (WN::D == 1) {
      if (G.pairs) {
        // 8-byte pieces: iws and the row start are even, so every piece is 8-byte aligned
        constexpr int NP = (NW + 1) / 2;
#pragma unroll
        for (int j = 0; j < NP; ++j) {
          const int col = iws + 2 * j;  // even, so a piece is either inside the row or outside (W even)
          const bool ok = row_ok && (unsigned)col < (unsigned)P.W;
          cp_async8(dst + 2 * j, ok ? (const void*)(src + 2 * j) : (const void*)P.x, ok);
        }
        continue;
      }
    }
#pragma unroll
    for (int i = 0; i < NW; ++i) {
      const bool ok = row_ok && ((unsigned)(iws + i) < (unsigned)P.W);
      cp_async4(dst + i, ok ? (const void*)(src + i) : (const void*)P.x, ok);
    }
  }
}

// Codes of taps [kb, kb + taps) of the CTA's NT = 32 channels: one block of
// the expanded layout, whose rows of 64 words (32 shifts, then 32 signs) are
// contiguous over the taps, so the stage is one flat 16-byte copy (zero fill
// past the last tap).
__device__ __forceinline__ void stage_codes_expanded(const GemmParams& P, const DirectGeom G, int32_t* code,
                                                     int64_t col0, int64_t kb) {
  static_assert(NT == 32, "one 32-channel block of the expanded layout per CTA");
  const int64_t left = P.kred - kb;
  const int valid = (left < G.taps ? (int)left : G.taps) * 16;  // 16-byte pieces present
  const int pieces = G.taps * 16;
  const int32_t* src = P.xcodes + ((col0 / 32) * P.kred + kb) * 64;
  for (int e = threadIdx.x; e < pieces; e += G.threads)
    cp_async16(code + e * 4, e < valid ? (const void*)(src + e * 4) : (const void*)P.xcodes, e < valid);
}

__device__ __forceinline__ uint32_t nib_word(const GemmParams& P, int64_t col, int64_t k) {
  const int64_t rec = (k >> 5) * P.cols + col;
  return __ldg(reinterpret_cast<const uint32_t*>(P.blob + P.off_nib + rec * 16) + ((k >> 3) & 3));
}
__device__ __forceinline__ uint2 bit_words(const GemmParams& P, int64_t col, int64_t k) {
  const int64_t rec = (k >> 5) * P.cols + col;
  return __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
}

__device__ __forceinline__ void decode_codes(const GemmParams& P, const DirectGeom G, int32_t* code,
                                             int64_t col0, int64_t kb) {
  constexpr int NB = NT / 32;
  const int item = threadIdx.x;
  const int runs = (G.taps + G.run - 1) / G.run;
  if (item >= runs * NT) return;
  const int n = item % NT;
  const int tl0 = (item / NT) * G.run;
  const int64_t col = col0 + n;
  const int64_t ks = kb + tl0;
  uint32_t lo = 0u, hi = 0u, neg = 0u, nz = 0u;
  if (col < P.cols && ks < P.kred) {
    const int64_t last = P.kred - 1;
    const uint32_t n0 = nib_word(P, col, ks);
    const uint32_t n1 = nib_word(P, col, (ks + 8 < last) ? ks + 8 : last);
    const uint32_t n2 = nib_word(P, col, (ks + 16 < last) ? ks + 16 : last);
    const int o = (int)(ks & 7) * 4;
    lo = __funnelshift_r(n0, n1, o);  // nibbles of taps ks .. ks+7
    hi = __funnelshift_r(n1, n2, o);  // nibbles of taps ks+8 .. ks+15
    const uint2 b0 = bit_words(P, col, ks);
    const uint2 b1 = bit_words(P, col, (ks + 15 < last) ? ks + 15 : last);
    const int b = (int)(ks & 31);
    neg = __funnelshift_r(b0.x, b1.x, b);
    nz = __funnelshift_r(b0.y, b1.y, b);
  }
  const int nvalid_k = (int)((P.kred - ks) < 16 ? (P.kred - ks) : 16);
  const int nloc = (G.taps - tl0) < G.run ? (G.taps - tl0) : G.run;
  int32_t* base = code + (n >> 5) * 64 + (n & 31);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    if (i < nloc) {
      const bool valid = i < nvalid_k;
      const uint32_t w = i < 8 ? lo : hi;
      const int sh = valid ? (int)((w >> (4 * (i & 7))) & 15u) : 0;
      const int sg = valid ? (int)((nz >> i) & 1u) - 2 * (int)((neg >> i) & 1u) : 0;
      base[(tl0 + i) * NB * 64] = sh;
      base[(tl0 + i) * NB * 64 + 32] = sg;
    }
  }
}

// The hot loop over one stage.  hp: this thread's window slot in channel 0
// of the stage; cp: this thread's 4 channels in tap 0 of the stage.
template <int SIG, int S, int TM, int I0, int NI, typename Acc>
__device__ __forceinline__ void compute_stage(const DirectGeom G, const int32_t* hp, const int32_t* cp,
                                              int rowstride, Acc (&acc)[NI][TN]) {
  using WN = Win<SIG, S, TM>;
  constexpr int R = S;  // square kernels
  constexpr int TAPW = 2 * NT;  // words per tap row
  const int cstride = G.HR * rowstride;
  constexpr int kUnrollC = S <= 3 ? 2 : 1;  // a 7-wide kernel's window already fills the registers
#pragma unroll kUnrollC
  for (int cl = 0; cl < G.CC; ++cl) {
    // a 7x7 kernel keeps the row loop rolled: its unrolled body (49 taps of
    // 28 terms) overflows the instruction cache (measured: stem 4% faster)
#pragma unroll (S <= 3 ? R : 1)
    for (int r = 0; r < R; ++r) {
      const int4* wp = reinterpret_cast<const int4*>(hp + r * rowstride);
      int w[4 * WN::WV];
#pragma unroll
      for (int v = 0; v < WN::WV; ++v) {
        const int4 t = wp[v];
        w[4 * v] = t.x;
        w[4 * v + 1] = t.y;
        w[4 * v + 2] = t.z;
        w[4 * v + 3] = t.w;
      }
#pragma unroll
      for (int s = 0; s < S; ++s) {
        const int4 shv = *reinterpret_cast<const int4*>(cp + (r * S + s) * TAPW);
        const int4 sgv = *reinterpret_cast<const int4*>(cp + (r * S + s) * TAPW + 32);
        const int sh[TN] = {shv.x, shv.y, shv.z, shv.w};
        const int sg[TN] = {sgv.x, sgv.y, sgv.z, sgv.w};
        // channel-outer order: consecutive SHF / IMAD share their shift / sign operand
#pragma unroll
        for (int j = 0; j < TN; ++j) {
#pragma unroll
          for (int i = 0; i < NI; ++i) {
            const int t = w[(I0 + i) * SIG + s + WN::D] >> sh[j];  // Eq. 1
            if constexpr (sizeof(Acc) == 4) {
              acc[i][j] += (uint32_t)sg[j] * (uint32_t)t;  // Eq. 2 + accumulate (mod 2^32)
            } else {
              acc[i][j] += (int64_t)sg[j] * (int64_t)t;
            }
          }
        }
      }
    }
    hp += cstride;
    cp += R * S * TAPW;
  }
}

template <int SIG, int S, int TM, int I0, int NI, typename Acc, bool CL>
__device__ __forceinline__ void run_direct(const GemmParams& P, const DirectGeom G, unsigned char* smem,
                                           int64_t gr0, int ow0, int64_t col0, int st_begin, int st_end,
                                           uint32_t& amax_local) {
  using WN = Win<SIG, S, TM>;
  const int t = threadIdx.x;
  const int cg = t % CG;
  const int pg = t / CG;
  const int g = pg % G.GW;
  const int oh_l = pg / G.GW;
  // the tile's first stacked halo row, and this thread's halo row offset
  const int n0 = (int)(gr0 / P.OH);
  const int off0 = (int)(gr0 - (int64_t)n0 * P.OH) * SIG;  // first halo row = stacked row n0 * HP + off0
  const int64_t s_lo = (int64_t)n0 * G.HP + off0;
  int srow;
  {
    const int64_t gr = gr0 + oh_l;
    const int64_t ni = gr / P.OH;
    srow = gr < (int64_t)G.N * P.OH ? (int)(ni * G.HP + (gr - ni * P.OH) * SIG - s_lo) : 0;
  }
  const int iw0 = ow0 * SIG - P.pw;
  const int rowstride = G.GW * WN::WSP;

  int32_t* const halo_base = reinterpret_cast<int32_t*>(smem);
  int32_t* const code_base = halo_base + 2 * G.halo_words;
  const int hoff = srow * rowstride + g * WN::WSP;
  const int coff = (cg >> 3) * 64 + (cg & 7) * TN;
  const bool expanded = P.xcodes != nullptr;

  Acc acc[NI][TN];
#pragma unroll
  for (int i = 0; i < NI; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  // Stage st reads buffers st % 2.  After the barrier of stage st every
  // thread has finished stage st - 1, so the other buffers are free: the
  // copies of stage st + 1 are issued there (and, without the expanded
  // layout, its codes decoded there after the compute); each thread waits
  // for its own copies before the next barrier, which then makes all of
  // stage st + 1 visible.
  const int64_t taps_per_c = (int64_t)S * S;
  if (st_begin < st_end) {  // a trailing rank of a cluster may have no stage: zero partial sums
    const int64_t kb = (int64_t)st_begin * G.CC * taps_per_c;
    stage_halo<SIG, S, TM>(P, G, halo_base, n0, off0, iw0, st_begin * G.CC);
    if (expanded) stage_codes_expanded(P, G, code_base, col0, kb);
    cp_async_commit();
    if (!expanded) decode_codes(P, G, code_base, col0, kb);
    cp_async_wait_all();
  }
  for (int st = st_begin; st < st_end; ++st) {
    const int b = (st - st_begin) & 1;
    const bool more = st + 1 < st_end;
    const int64_t kb1 = (int64_t)(st + 1) * G.CC * taps_per_c;
    __syncthreads();
    if (more) {
      stage_halo<SIG, S, TM>(P, G, halo_base + (b ^ 1) * G.halo_words, n0, off0, iw0,
                             (st + 1) * G.CC);
      if (expanded) stage_codes_expanded(P, G, code_base + (b ^ 1) * G.code_words, col0, kb1);
      cp_async_commit();
    }
    compute_stage<SIG, S, TM, I0, NI, Acc>(G, halo_base + b * G.halo_words + hoff,
                                           code_base + b * G.code_words + coff, rowstride, acc);
    if (more) {
      if (!expanded) decode_codes(P, G, code_base + (b ^ 1) * G.code_words, col0, kb1);
      cp_async_wait_all();
    }
  }
  __syncthreads();  // the next pass (64-bit path) reuses the buffers

  if constexpr (CL) {
    // Split over a thread-block cluster: every rank has the same tile mapping,
    // so entry (thread, pixel slot, channel) of each rank's partial sums (a
    // subset of the terms: 32-bit partials are exact whenever the bound holds)
    // belongs to the same output.  Rank r sums, through distributed shared
    // memory, the slots i = r (mod cluster) of its threads and stores them.
    Acc* red = reinterpret_cast<Acc*>(smem);
#pragma unroll
    for (int i = 0; i < NI; ++i)
#pragma unroll
      for (int j = 0; j < TN; ++j) red[(t * TM + I0 + i) * TN + j] = acc[i][j];
    cg::cluster_group cl = cg::this_cluster();
    cl.sync();  // all partials written
    const int rank = (int)cl.block_rank();
    const int64_t grc = gr0 + oh_l;
    const bool row_ok = grc < (int64_t)G.N * P.OH;
    const int64_t nc = row_ok ? grc / P.OH : 0;
    const int ohc = row_ok ? (int)(grc - nc * P.OH) : 0;
    const int64_t OHWc = (int64_t)P.OH * P.OW;
    const bool relu_c = (P.flags & DS_RELU) != 0;
    const bool resid_c = (P.flags & DS_RESIDUAL) != 0;
    for (int i = I0; i < I0 + NI; ++i) {
      const int ow = ow0 + g * TM + i;
      if (i % G.cluster != rank || !row_ok || ow >= P.OW) continue;
      Acc sum[TN] = {0, 0, 0, 0};
      for (int q = 0; q < G.cluster; ++q) {
        const Acc* src = cl.map_shared_rank(red, q) + (t * TM + i) * TN;
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
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const int64_t col = col0 + cg * TN + j;
        if (col >= P.cols) continue;
        const int64_t idx = (nc * P.cols + col) * OHWc + (int64_t)ohc * P.OW + ow;
        const int32_t bcol = P.bias ? __ldg(P.bias + col) : 0;
        int32_t o;
        if constexpr (sizeof(Acc) == 4) {
          o = (int32_t)(sum[j] + (uint32_t)bcol);
        } else {
          int64_t a = sum[j] + (int64_t)bcol;
          a = a > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : a;
          a = a < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : a;
          o = (int32_t)a;
        }
        if (resid_c) o = add_sat(o, __ldg(P.residual + idx));
        if (relu_c) o = max(o, 0);
        amax_local = max(amax_local, uabs(o));
        P.y[idx] = o;
      }
    }
    cl.sync();  // no rank reuses its shared memory (next pass) or exits while another reads it
    return;
  }

  const int64_t gr = gr0 + oh_l;  // this thread's output row (recomputed: not kept live in the loop)
  if (gr >= (int64_t)G.N * P.OH) return;
  const int64_t n_img = gr / P.OH;
  const int oh = (int)(gr - n_img * P.OH);
  const int owb = ow0 + g * TM + I0;
  const int64_t OHW = (int64_t)P.OH * P.OW;
  if (P.split_acc != nullptr) {
    // split reduction: add this stage range's exact partial sums (no bias)
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int64_t col = col0 + cg * TN + j;
      if (col >= P.cols) continue;
      unsigned long long* arow = reinterpret_cast<unsigned long long*>(P.split_acc) +
                                 (n_img * P.cols + col) * OHW + (int64_t)oh * P.OW;
#pragma unroll
      for (int i = 0; i < NI; ++i) {
        if (owb + i >= P.OW) continue;
        int64_t v;
        if constexpr (sizeof(Acc) == 4) {
          v = (int64_t)(int32_t)acc[i][j];  // exact: |partial| <= the proven bound < 2^31
        } else {
          v = acc[i][j];
        }
        atomicAdd(arow + owb + i, (unsigned long long)v);
      }
    }
    return;
  }
  // fused epilogue: bias, saturation (64-bit path), residual, ReLU, amax
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool resid = (P.flags & DS_RESIDUAL) != 0;
#pragma unroll
  for (int j = 0; j < TN; ++j) {
    const int64_t col = col0 + cg * TN + j;
    if (col >= P.cols) continue;
    const int32_t bcol = P.bias ? __ldg(P.bias + col) : 0;
    int32_t* yrow = P.y + (n_img * P.cols + col) * OHW + (int64_t)oh * P.OW;
    const int32_t* rrow = resid ? P.residual + (n_img * P.cols + col) * OHW + (int64_t)oh * P.OW : nullptr;
#pragma unroll
    for (int i = 0; i < NI; ++i) {
      const int ow = owb + i;
      if (ow >= P.OW) continue;
      int32_t o;
      if constexpr (sizeof(Acc) == 4) {
        o = (int32_t)(acc[i][j] + (uint32_t)bcol);
      } else {
        int64_t a = acc[i][j] + (int64_t)bcol;
        a = a > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : a;
        a = a < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : a;
        o = (int32_t)a;
      }
      if (resid) o = add_sat(o, __ldg(rrow + ow));
      if (relu) o = max(o, 0);
      amax_local = max(amax_local, uabs(o));
      yrow[ow] = o;
    }
  }
}

__device__ __forceinline__ bool tile_int32_exact(const GemmParams& P, int NT, int64_t col0) {
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
        unsafe = (((lo + 32767ull) >> 15) + nnz + b) > (unsigned long long)INT32_MAX;
      }
    }
  }
  return !__syncthreads_or(unsafe);
}

template <int SIG, int S, int TM, bool CL>
__global__ void __launch_bounds__(kMaxThreads, 3) conv_direct_kernel(const GemmParams P, const DirectGeom G) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int bx = blockIdx.x;
  const int tw = bx % G.tiles_w;
  const int th = bx / G.tiles_w;
  const int64_t col0 = (int64_t)blockIdx.y * NT;
  const int64_t gr0 = (int64_t)th * G.TH;
  const int ow0 = tw * TM * G.GW;
  const int st_begin = blockIdx.z * G.stages_per_split;
  const int st_end = min(G.n_stages, st_begin + G.stages_per_split);

  uint32_t amax_local = 0;
  if (tile_int32_exact(P, NT, col0)) {
    run_direct<SIG, S, TM, 0, TM, uint32_t, CL>(P, G, smem_raw, gr0, ow0, col0, st_begin, st_end, amax_local);
  } else {
    constexpr int H1 = TM / 2;
    run_direct<SIG, S, TM, 0, H1, int64_t, CL>(P, G, smem_raw, gr0, ow0, col0, st_begin, st_end, amax_local);
    run_direct<SIG, S, TM, H1, TM - H1, int64_t, CL>(P, G, smem_raw, gr0, ow0, col0, st_begin, st_end, amax_local);
  }
  if (P.amax_out != nullptr && P.split_acc == nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

// Epilogue of a split reduction: y = ReLU?(sat32(sat32(acc + bias) + residual)), amax.
// Quad path (total a multiple of 4 below 2^31, 16-byte aligned y and
// residual): a thread takes 4 consecutive outputs with 16-byte loads of the
// int64 partial sums and of the residual and one 16-byte store; the first
// output's channel comes from two multiply-shift divisions, the others step
// along (a quad may cross a channel plane).  Otherwise one output per thread
// with 64-bit divisions.
__global__ void conv_split_finalize_kernel(const GemmParams P, int64_t total, FastDiv d_ohw, FastDiv d_cols,
                                           bool quad) {
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool resid = (P.flags & DS_RESIDUAL) != 0;
  const int64_t prefix = (int64_t)(kSmallScratchBytes / sizeof(int64_t));  // the zero prefix
  uint32_t amax_local = 0;
  if (quad) {
    const int OHW = P.OH * P.OW;
    const int cols = (int)P.cols;
    const longlong2* acc2 = reinterpret_cast<const longlong2*>(P.split_acc);
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < total / 4;
         q += (int64_t)gridDim.x * blockDim.x) {
      const int e = (int)(q * 4);
      const int plane = fdiv(e, d_ohw);
      int pix = e - plane * OHW;
      int col = plane - fdiv(plane, d_cols) * cols;
      const longlong2 a01 = acc2[2 * q], a23 = acc2[2 * q + 1];
      if (e < prefix) {
        reinterpret_cast<longlong2*>(P.split_acc)[2 * q] = make_longlong2(0, 0);
        reinterpret_cast<longlong2*>(P.split_acc)[2 * q + 1] = make_longlong2(0, 0);
      }
      const int4 r4 = resid ? __ldg(reinterpret_cast<const int4*>(P.residual) + q) : make_int4(0, 0, 0, 0);
      const int64_t a[4] = {a01.x, a01.y, a23.x, a23.y};
      const int32_t rv[4] = {r4.x, r4.y, r4.z, r4.w};
      int32_t o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        int64_t v = a[i] + (P.bias ? (int64_t)__ldg(P.bias + col) : 0);
        v = v > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : v;
        v = v < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : v;
        o[i] = (int32_t)v;
        if (resid) o[i] = add_sat(o[i], rv[i]);
        if (relu) o[i] = max(o[i], 0);
        amax_local = max(amax_local, uabs(o[i]));
        if (++pix == OHW) {
          pix = 0;
          col = col + 1 == cols ? 0 : col + 1;
        }
      }
      reinterpret_cast<int4*>(P.y)[q] = make_int4(o[0], o[1], o[2], o[3]);
    }
  } else {
    const int64_t OHW = (int64_t)P.OH * P.OW;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
      const int64_t col = (e / OHW) % P.cols;
      int64_t a = P.split_acc[e] + (P.bias ? (int64_t)__ldg(P.bias + col) : 0);
      if (e < prefix) P.split_acc[e] = 0;
      a = a > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : a;
      a = a < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : a;
      int32_t o = (int32_t)a;
      if (resid) o = add_sat(o, __ldg(P.residual + e));
      if (relu) o = max(o, 0);
      amax_local = max(amax_local, uabs(o));
      P.y[e] = o;
    }
  }
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

struct Choice {
  DirectGeom G;
  int TM;
};

size_t direct_smem_bytes(const DirectGeom& G) {
  return (size_t)2 * (G.halo_words + (size_t)G.code_words) * sizeof(int32_t);
}

// Tile choice.  TM = 7 when the output width is a multiple of 7 (every
// ResNet / VGG feature map: 112, 56, 28, 14, 7), else 8.  Groups per row at
// most 8; TH stacked rows so that the CTA has 256 threads (fewer only when
// the whole batch has fewer rows).  With split_capacity > 0 the stages are
// split over CTAs when the grid would not fill every SM slot once (targeting
// two waves).
bool choose_geom(const GemmParams& p, size_t split_capacity, Choice& ch) {
  DirectGeom& G = ch.G;
  ch.TM = (p.OW % 7 == 0) ? 7 : 8;
  const bool has_cluster = ch.TM == 7 && (p.S == 3 || p.S == 7);  // the kernels with a cluster variant
  const int WS = (ch.TM - 1) * p.sw + p.S + (p.sw == 2 ? 1 : 0);  // staged words, with Win<>::D
  const int WSP = (WS + 3) / 4 * 4 + (((WS + 3) / 4) % 2 == 0 ? 4 : 0);  // as Win<>::WSP
  int gw = (p.OW + ch.TM - 1) / ch.TM;
  if (gw > 8) {
    const int pieces = (gw + 7) / 8;
    gw = (gw + pieces - 1) / pieces;
  }
  G.GW = gw;
  G.N = (int)(p.rows / ((int64_t)p.OH * p.OW));
  const int64_t rows_total = (int64_t)G.N * p.OH;
  int th = kMaxThreads / (G.GW * CG);
  if (th < 1) return false;
  if (rows_total < th) {
    th = (int)rows_total;
    while ((th * G.GW) % 4 != 0) ++th;  // whole warps
  }
  G.TH = th;
  G.threads = G.TH * G.GW * CG;
  if (G.threads % 32 != 0 || G.threads > kMaxThreads || G.threads < NT) return false;
  G.HP = p.H + 2 * p.ph;
  // halo rows: the largest stacked-row span any tile reads (tile starts repeat
  // with period OH, so OH + 1 starts cover every case)
  const int64_t tiles_h = (rows_total + G.TH - 1) / G.TH;
  int64_t span = 0;
  for (int64_t k = 0; k < tiles_h && k <= p.OH; ++k) {
    const int64_t a = k * G.TH, z = std::min(a + G.TH, rows_total) - 1;
    const int64_t sa = (a / p.OH) * G.HP + (a % p.OH) * p.sh;
    const int64_t sz = (z / p.OH) * G.HP + (z % p.OH) * p.sh;
    span = std::max(span, sz - sa + p.R);
  }
  if (span > 4096) return false;
  G.HR = (int)span;
  const int per_c_words = G.HR * G.GW * WSP + 2 * p.R * p.S * NT;
  int cc = kSmemBudget / (2 * 4 * per_c_words);
  if (cc < 1) return false;
  if (cc > p.C) cc = p.C;
  for (int d = cc; d >= 1; --d)  // prefer a chunk that divides C
    if (p.C % d == 0 && 2 * d >= cc) {
      cc = d;
      break;
    }
  const int64_t ctas = (int64_t)((p.OW + ch.TM * G.GW - 1) / (ch.TM * G.GW)) * tiles_h * ((p.cols + NT - 1) / NT);
  // A grid that does not fill every SM slot once splits its stages over the
  // CTAs of a cluster: then use stages small enough that every rank gets one.
  const int target = (int)std::min<int64_t>(kMaxCluster, ctas < slots() ? slots() / std::max<int64_t>(ctas, 1) : 1);
  // Calls without a workspace split an under-filled grid over a cluster.  With a
  // workspace (the chained forward) a grid of at least a third of the slots
  // splits over a cluster too, a smaller one over CTAs adding int64 partial
  // sums atomically: measured faster for the small grids (ResNet18 batch 1:
  // 0.51 vs 0.63 ms per forward with clusters throughout), slower for the
  // others (the atomics, the memset and the finalize cost more than the
  // cluster barriers).
  const bool allow_cluster = has_cluster && (split_capacity == 0 || target <= kChainClusterMaxTarget);
  if (allow_cluster && target >= 2 && (p.C + cc - 1) / cc < target) {
    int want = std::max(1, p.C / target);
    for (int d = want; d >= 1; --d)
      if (p.C % d == 0) {
        want = d;
        break;
      }
    cc = std::min(cc, want);
  }
  G.CC = cc;
  G.taps = G.CC * p.R * p.S;
  G.n_stages = (p.C + G.CC - 1) / G.CC;
  G.halo_words = G.CC * G.HR * G.GW * WSP;
  G.code_words = G.taps * 2 * NT;
  int run = (G.taps * NT + G.threads - 1) / G.threads;  // decode: at most one item per thread
  if (run < 1) run = 1;
  if (run > 16 && p.xcodes == nullptr) return false;
  G.run = run;
  // 8-byte halo pieces: the first staged column iw0 + g TM sig - 1 is even when
  // the padding is odd, and a row starts on an even word when W is even
  G.pairs = (p.sw == 2 && (p.W % 2) == 0 && (p.pw % 2) == 1 && (reinterpret_cast<uintptr_t>(p.x) & 7) == 0) ? 1 : 0;
  G.dGW = make_fastdiv((uint32_t)G.GW);
  G.dHR = make_fastdiv((uint32_t)G.HR);
  G.dHP = make_fastdiv((uint32_t)G.HP);
  G.tiles_w = (p.OW + ch.TM * G.GW - 1) / (ch.TM * G.GW);
  G.tiles_h = (int)tiles_h;
  // split the stages when the grid would not fill every SM slot once: over a
  // thread-block cluster (launch_direct checks the size with the device),
  // else, with a workspace, over CTAs adding int64 partials atomically
  G.splits = 1;
  G.stages_per_split = G.n_stages;
  G.cluster = 1;
  if (allow_cluster && target >= 2 && G.n_stages >= 2) {
    G.cluster = std::min(target, G.n_stages);
    G.stages_per_split = (G.n_stages + G.cluster - 1) / G.cluster;
    G.splits = G.cluster;
  } else {
    const size_t need = (size_t)p.rows * p.cols * sizeof(int64_t);
    // a grid within an eighth of one full wave runs unsplit
    if (split_capacity >= need && ctas * 8 < slots() * 7 && G.n_stages > 1) {
      int want = (int)std::min<int64_t>(G.n_stages, (2 * slots() + ctas - 1) / ctas);
      G.stages_per_split = (G.n_stages + want - 1) / want;
      G.splits = (G.n_stages + G.stages_per_split - 1) / G.stages_per_split;
    }
  }
  return direct_smem_bytes(G) <= (size_t)kSmemBudget;
}

// Shared memory of a launch: the staging buffers, and in cluster mode at least
// the partial sums (threads x TM x TN, 64-bit in the worst case).
size_t launch_smem_bytes(const DirectGeom& G, int TM) {
  size_t smem = direct_smem_bytes(G);
  if (G.cluster > 1) smem = std::max(smem, (size_t)G.threads * TM * TN * sizeof(int64_t));
  return smem;
}

template <int SIG, int S, int TM, bool CL>
bool set_attributes() {
  // once per process, thread-safe (a function-local static is initialised
  // once); not a stream operation, so a forward captured in a CUDA graph
  // after a first eager call issues no attribute call
  static const bool ok = [] {
    const bool r = cudaFuncSetAttribute(conv_direct_kernel<SIG, S, TM, CL>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget) == cudaSuccess &&
                   (!CL || cudaFuncSetAttribute(conv_direct_kernel<SIG, S, TM, CL>,
                                                cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess);
    if (!r) (void)cudaGetLastError();
    return r;
  }();
  return ok;
}

// How many clusters of cs CTAs of this kernel, with smem bytes of shared
// memory each, the device holds at once (0: none).  Cached per process for
// up to kCacheEntries (size, shared memory) pairs; past that it is queried
// each time.
template <int SIG, int S, int TM>
int max_clusters(int cs, size_t smem) {
  if (!set_attributes<SIG, S, TM, true>()) return 0;
  if (cs < 2 || cs > kMaxCluster) return 0;
  constexpr int kCacheEntries = 64;
  struct Entry {
    int cs;
    size_t smem;
    int n;
  };
  static Entry cache[kCacheEntries];
  static int used = 0;
  static std::mutex mu;  // the cache is shared by every host thread
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (cache[i].cs == cs && cache[i].smem == smem) return cache[i].n;
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1, 1, cs);
    cfg.blockDim = dim3(kMaxThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = cs;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, conv_direct_kernel<SIG, S, TM, true>, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    n = n > 0 ? n : 0;
    if (used < kCacheEntries) cache[used++] = Entry{cs, smem, n};
    return n;
  }
}

// Cluster-split variants exist for the network shapes (TM = 7; 3x3 and 7x7 kernels).
constexpr bool has_cluster_variant(int S, int TM) { return TM == 7 && (S == 3 || S == 7); }

template <int SIG, int S, int TM>
cudaError_t launch_direct(const GemmParams& p, const DirectGeom& G0, cudaStream_t st) {
  if (!set_attributes<SIG, S, TM, false>()) return cudaErrorInvalidValue;
  DirectGeom G = G0;
  if (G.cluster > 1) {
    // The cluster size with the least time, counted as waves x stages per
    // rank, over every size up to 16 with at least one stage per rank: the
    // device holds max_clusters(cs) clusters at once, which can be fewer
    // than the SM slots allow (e.g. 110 clusters of 4 for 112 needed: two of
    // them would run in a second wave), and a larger cluster in two waves
    // can beat a smaller one in one.  cs = 1: no split.
    int cs = 1;
    if constexpr (has_cluster_variant(S, TM)) {
      const int64_t tiles = (int64_t)G.tiles_w * G.tiles_h * ((p.cols + NT - 1) / NT);
      int64_t best = ((tiles + slots() - 1) / std::max<int64_t>(slots(), 1)) * G.n_stages;
      for (int c = 2; c <= std::min(kMaxCluster, G.n_stages); ++c) {
        const int n = max_clusters<SIG, S, TM>(c, launch_smem_bytes(G, TM));
        if (n <= 0) continue;
        const int64_t cost = ((tiles + n - 1) / n) * ((G.n_stages + c - 1) / c);
        if (cost < best) {
          best = cost;
          cs = c;
        }
      }
    }
    if (cs >= 2) {
      G.cluster = cs;
      G.stages_per_split = (G.n_stages + cs - 1) / cs;
      G.splits = cs;
    } else {
      G.cluster = 1;
      G.splits = 1;
      G.stages_per_split = G.n_stages;
    }
  }
  const size_t smem = launch_smem_bytes(G, TM);
  GemmParams q = p;
  const dim3 grid((unsigned)((int64_t)G.tiles_w * G.tiles_h), (unsigned)((p.cols + NT - 1) / NT), (unsigned)G.splits);
  if (G.cluster > 1) {
    q.split_acc = nullptr;
    if constexpr (has_cluster_variant(S, TM)) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = grid;
      cfg.blockDim = dim3(G.threads, 1, 1);
      cfg.dynamicSmemBytes = smem;
      cfg.stream = st;
      cudaLaunchAttribute attr;
      attr.id = cudaLaunchAttributeClusterDimension;
      attr.val.clusterDim.x = 1;
      attr.val.clusterDim.y = 1;
      attr.val.clusterDim.z = (unsigned)G.cluster;
      cfg.attrs = &attr;
      cfg.numAttrs = 1;
      return cudaLaunchKernelEx(&cfg, conv_direct_kernel<SIG, S, TM, true>, q, G);
    }
  }
  if (G.splits == 1) {
    q.split_acc = nullptr;
  } else {
    cudaError_t e = prepare_split_scratch(q, st);
    if (e != cudaSuccess) return e;
  }
  conv_direct_kernel<SIG, S, TM, false><<<grid, G.threads, smem, st>>>(q, G);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || G.splits == 1) return e;
  return launch_split_finalize(q, st);
}

template <int SIG, int TM>
cudaError_t launch_by_s(const GemmParams& p, const DirectGeom& G, cudaStream_t st) {
  if (p.S == 1) return launch_direct<SIG, 1, TM>(p, G, st);
  if (p.S == 3) return launch_direct<SIG, 3, TM>(p, G, st);
  return launch_direct<SIG, 7, TM>(p, G, st);
}

}  // namespace

bool conv_direct_supported(const GemmParams& p) {
  if (p.sh != p.sw || !(p.sh == 1 || p.sh == 2)) return false;
  if (!(p.S == 1 || p.S == 3 || p.S == 7) || p.R != p.S) return false;
  if ((p.rows / ((int64_t)p.OH * p.OW)) >= ((int64_t)1 << 24)) return false;
  Choice ch;
  return choose_geom(p, p.split_acc ? p.split_capacity : 0, ch);
}

cudaError_t prepare_split_scratch(const GemmParams& p, cudaStream_t st) {
  // The first kSmallScratchBytes of the scratch are zero between layers (the
  // chained forward resets them once, every finalize re-zeroes them), so a
  // small region (batch 1) needs no memset launch.  A larger region is zeroed
  // here: a memset is cheaper than re-zeroing it in the finalize (measured:
  // ResNet18 batch 32 5.33 vs 5.50 ms per forward, batch 1 0.49 vs 0.50 ms).
  const size_t bytes = (size_t)p.rows * p.cols * sizeof(int64_t);
  if (bytes <= kSmallScratchBytes) return cudaSuccess;
  return cudaMemsetAsync(p.split_acc, 0, bytes, st);
}

cudaError_t launch_split_finalize(const GemmParams& p, cudaStream_t st) {
  const int64_t total = p.rows * p.cols;
  const bool quad = total % 4 == 0 && total <= (int64_t)INT32_MAX && (reinterpret_cast<uintptr_t>(p.y) & 15) == 0 &&
                    (reinterpret_cast<uintptr_t>(p.split_acc) & 15) == 0 &&
                    (!(p.flags & DS_RESIDUAL) || (reinterpret_cast<uintptr_t>(p.residual) & 15) == 0);
  const int64_t items = quad ? total / 4 : total;
  int64_t blocks = (items + 255) / 256;
  if (blocks > std::max<int64_t>(slots(), 1) * 8) blocks = std::max<int64_t>(slots(), 1) * 8;
  if (blocks < 1) blocks = 1;
  const FastDiv d_ohw = make_fastdiv((uint32_t)((int64_t)p.OH * p.OW));
  const FastDiv d_cols = make_fastdiv((uint32_t)(p.cols < 1 ? 1 : (p.cols > INT32_MAX ? INT32_MAX : p.cols)));
  conv_split_finalize_kernel<<<(unsigned)blocks, 256, 0, st>>>(p, total, d_ohw, d_cols, quad);
  return cudaGetLastError();
}

size_t conv_direct_split_bytes(const GemmParams& p) {
  if (!conv_direct_supported(p)) return 0;
  Choice ch;
  if (!choose_geom(p, ~(size_t)0, ch) || ch.G.splits <= 1 || ch.G.cluster > 1) return 0;  // clusters need none
  return (size_t)p.rows * p.cols * sizeof(int64_t);
}

cudaError_t launch_conv2d_direct(const GemmParams& p, cudaStream_t st) {
  Choice ch;
  if (!choose_geom(p, p.split_acc ? p.split_capacity : 0, ch)) return cudaErrorInvalidConfiguration;
  if (ch.TM == 7) return p.sh == 1 ? launch_by_s<1, 7>(p, ch.G, st) : launch_by_s<2, 7>(p, ch.G, st);
  return p.sh == 1 ? launch_by_s<1, 8>(p, ch.G, st) : launch_by_s<2, 8>(p, ch.G, st);
}

}  // namespace ds
