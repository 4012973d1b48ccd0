// ConvShift forward, direct (halo-tile) kernel (DeepShift Eq. 1-3, Sec. 4).
//
//   y[n][k][oh][ow] = sat32( b[k] + sum_{c,r,s} s_w * (xpad[n][c][oh*sig + r][ow*sig + s] >> -p) )
//
// Each CTA owns one image, TH output rows x TW = 8*GW output columns and 64
// output channels.  The input rows and columns that tile reads (its halo,
// zero outside the image) are staged into shared memory once per chunk of
// input channels with cp.async; the decoded codes of the same chunk (shift
// and sign as 32-bit words, one row per tap) are staged next to them.  A
// thread owns 8 consecutive output pixels of one row and TN channels.  For
// each (c, r) it loads one window of 7*sig + S input values from the halo
// row into registers and reuses it for all S taps of that row (sliding
// window), so the hot loop is, per term, one arithmetic right shift (ALU
// pipe) and one multiply-add by the sign (FMA pipe) with no im2col copy.
//
// Accumulator width as in shift_gemm.cu: 32-bit when the launch bound proves
// it exact for the CTA's channels, else a 64-bit pass per half of the pixels.
#include "ds_common.cuh"

namespace ds {
namespace {

constexpr int NT = 64;  // output channels per CTA
constexpr int TM = 8;   // output pixels per thread (consecutive ow)
constexpr int TN = 4;   // output channels per thread
constexpr int CG = NT / TN;  // channel groups per CTA (16)
constexpr int kMaxThreads = 224;  // 3 CTAs per SM at <= 96 registers

struct DirectGeom {
  int TH, GW;      // output rows and 8-column groups per CTA
  int CC;          // input channels per stage
  int HR, HWP;     // halo rows, halo row stride (words)
  int taps;        // CC * R * S
  int n_stages;    // ceil(C / CC)
  int halo_words;  // CC * HR * HWP
  int code_words;  // taps * NT
  int threads;     // TH * GW * CG
};

__device__ __forceinline__ void cp_async4(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  const int n = valid ? 4 : 0;
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(gsrc), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}
__device__ __forceinline__ int32_t add_sat(int32_t a, int32_t b) {
  int32_t r;
  asm("add.sat.s32 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t uabs(int32_t v) {
  return v < 0 ? (uint32_t)0 - (uint32_t)v : (uint32_t)v;
}

// Stage the halo of input channels [c0, c0 + CC) for this CTA.  One warp per
// halo row, lanes along the row; zero outside the image and beyond C.
__device__ __forceinline__ void stage_halo(const GemmParams& P, const DirectGeom G, int32_t* halo,
                                           int64_t img_base, int ih0, int iw0, int c0, int HWd) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = G.threads >> 5;
  const int64_t HW = (int64_t)P.H * P.W;
  for (int row = warp; row < G.CC * G.HR; row += nwarps) {
    const int cl = row / G.HR;
    const int hr = row - cl * G.HR;
    const int c = c0 + cl;
    const int ih = ih0 + hr;
    const bool row_ok = (c < P.C) && ((unsigned)ih < (unsigned)P.H);
    const int32_t* src_row = P.x + img_base + (int64_t)c * HW + (int64_t)ih * P.W;
    int32_t* dst_row = halo + row * G.HWP;
    for (int hc = lane; hc < HWd; hc += 32) {
      const int iw = iw0 + hc;
      const bool ok = row_ok && ((unsigned)iw < (unsigned)P.W);
      cp_async4(dst_row + hc, ok ? (const void*)(src_row + iw) : (const void*)P.x, ok);
    }
  }
}

// Decode the codes of taps [kb, kb + taps) for the CTA's 64 channels into
// shift / sign words.  Work item = (channel, run of 8 taps).
__device__ __forceinline__ uint32_t nib_word(const GemmParams& P, int64_t col, int64_t k) {
  const int64_t rec = (k >> 5) * P.cols + col;
  return __ldg(reinterpret_cast<const uint32_t*>(P.blob + P.off_nib + rec * 16) + ((k >> 3) & 3));
}
__device__ __forceinline__ uint2 bit_words(const GemmParams& P, int64_t col, int64_t k) {
  const int64_t rec = (k >> 5) * P.cols + col;
  return __ldg(reinterpret_cast<const uint2*>(P.blob + P.off_bits + rec * 8));
}

__device__ __forceinline__ void stage_codes(const GemmParams& P, const DirectGeom G, int32_t* sh_s,
                                            int32_t* sg_s, int64_t col0, int64_t kb) {
  const int runs = (G.taps + 7) >> 3;
  for (int item = threadIdx.x; item < runs * NT; item += G.threads) {
    const int n = item & (NT - 1);
    const int q = item >> 6;
    const int64_t col = col0 + n;
    const int64_t ks = kb + 8 * q;
    const int tl0 = 8 * q;  // local tap index of ks
    uint32_t nib = 0u, neg = 0u, nz = 0u;
    if (col < P.cols && ks < P.kred) {
      const int64_t khi = (ks + 8 < P.kred) ? ks + 8 : P.kred - 1;
      const uint32_t lo = nib_word(P, col, ks);
      const uint32_t hi = nib_word(P, col, khi);
      nib = __funnelshift_r(lo, hi, 4 * (int)(ks & 7));
      const int64_t kb2 = (ks + 7 < P.kred) ? ks + 7 : P.kred - 1;
      const uint2 blo = bit_words(P, col, ks);
      const uint2 bhi = bit_words(P, col, kb2);
      neg = __funnelshift_r(blo.x, bhi.x, (int)(ks & 31));
      nz = __funnelshift_r(blo.y, bhi.y, (int)(ks & 31));
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int tl = tl0 + i;
      if (tl < G.taps) {
        const bool valid = (ks + i) < P.kred;
        const int sh = valid ? (int)((nib >> (4 * i)) & 15u) : 0;
        const int sg = valid ? (int)((nz >> i) & 1u) - 2 * (int)((neg >> i) & 1u) : 0;
        sh_s[tl * NT + n] = sh;
        sg_s[tl * NT + n] = sg;
      }
    }
  }
}

// The hot loop over one stage: for every (c, r) one window load, then S taps
// of 8 pixels x TN channels, two instructions per term.
template <int SIG, int S, int I0, int NI, typename Acc>
__device__ __forceinline__ void compute_stage(const GemmParams& P, const DirectGeom G,
                                              const int32_t* halo, const int32_t* sh_s,
                                              const int32_t* sg_s, int oh_l, int g, int cg,
                                              Acc (&acc)[NI][TN]) {
  constexpr int WS = 7 * SIG + S;          // window values used
  constexpr int WV = (WS + 3) / 4;         // 16-byte loads per window
  const int32_t* hbase = halo + (oh_l * SIG) * G.HWP + g * 8 * SIG;
  const int32_t* shb = sh_s + cg * TN;
  const int32_t* sgb = sg_s + cg * TN;
  for (int cl = 0; cl < G.CC; ++cl) {
    for (int r = 0; r < P.R; ++r) {
      const int4* wp = reinterpret_cast<const int4*>(hbase + (cl * G.HR + r) * G.HWP);
      int w[4 * WV];
#pragma unroll
      for (int v = 0; v < WV; ++v) {
        const int4 t = wp[v];
        w[4 * v] = t.x;
        w[4 * v + 1] = t.y;
        w[4 * v + 2] = t.z;
        w[4 * v + 3] = t.w;
      }
      const int tap0 = (cl * P.R + r) * S;
#pragma unroll
      for (int s = 0; s < S; ++s) {
        const int4 shv = *reinterpret_cast<const int4*>(shb + (tap0 + s) * NT);
        const int4 sgv = *reinterpret_cast<const int4*>(sgb + (tap0 + s) * NT);
        const int sh[TN] = {shv.x, shv.y, shv.z, shv.w};
        const int sg[TN] = {sgv.x, sgv.y, sgv.z, sgv.w};
#pragma unroll
        for (int i = 0; i < NI; ++i) {
          const int xv = w[(I0 + i) * SIG + s];
#pragma unroll
          for (int j = 0; j < TN; ++j) {
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
  }
}

template <int SIG, int S, int I0, int NI, typename Acc>
__device__ __forceinline__ void run_direct(const GemmParams& P, const DirectGeom G, unsigned char* smem,
                                           int n_img, int oh0, int ow0, int64_t col0,
                                           uint32_t& amax_local) {
  const int t = threadIdx.x;
  const int cg = t % CG;
  const int pg = t / CG;
  const int g = pg % G.GW;
  const int oh_l = pg / G.GW;
  const int HWd = (8 * G.GW - 1) * SIG + S;
  const int64_t img_base = (int64_t)n_img * P.C * P.H * P.W;
  const int ih0 = oh0 * SIG - P.ph;
  const int iw0 = ow0 * SIG - P.pw;

  int32_t* const smem_base = reinterpret_cast<int32_t*>(smem);
  const int stage_words = G.halo_words + 2 * G.code_words;

  Acc acc[NI][TN];
#pragma unroll
  for (int i = 0; i < NI; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0;

  const int64_t taps_per_c = (int64_t)P.R * S;
  stage_halo(P, G, smem_base, img_base, ih0, iw0, 0, HWd);
  cp_async_commit();
  stage_codes(P, G, smem_base + G.halo_words, smem_base + G.halo_words + G.code_words, col0, 0);
  for (int st = 0; st < G.n_stages; ++st) {
    int32_t* const cur = smem_base + (st & 1) * stage_words;
    int32_t* const nxt = smem_base + ((st & 1) ^ 1) * stage_words;
    if (st + 1 < G.n_stages) {
      const int c1 = (st + 1) * G.CC;
      stage_halo(P, G, nxt, img_base, ih0, iw0, c1, HWd);
      cp_async_commit();
      stage_codes(P, G, nxt + G.halo_words, nxt + G.halo_words + G.code_words, col0,
                  (int64_t)c1 * taps_per_c);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    compute_stage<SIG, S, I0, NI, Acc>(P, G, cur, cur + G.halo_words, cur + G.halo_words + G.code_words,
                                       oh_l, g, cg, acc);
    __syncthreads();
  }

  // fused epilogue: bias, saturation (64-bit path), residual, ReLU, amax
  const int oh = oh0 + oh_l;
  if (oh >= P.OH) return;
  const bool relu = (P.flags & DS_RELU) != 0;
  const bool resid = (P.flags & DS_RESIDUAL) != 0;
  const int owb = ow0 + g * 8 + I0;
  const int64_t OHW = (int64_t)P.OH * P.OW;
#pragma unroll
  for (int j = 0; j < TN; ++j) {
    const int64_t col = col0 + cg * TN + j;
    if (col >= P.cols) continue;
    const int32_t bcol = P.bias ? __ldg(P.bias + col) : 0;
    const int64_t rowbase = ((int64_t)n_img * P.cols + col) * OHW + (int64_t)oh * P.OW;
    int32_t v[NI];
#pragma unroll
    for (int i = 0; i < NI; ++i) {
      if constexpr (sizeof(Acc) == 4) {
        v[i] = (int32_t)(acc[i][j] + (uint32_t)bcol);
      } else {
        int64_t a = acc[i][j] + (int64_t)bcol;
        a = a > (int64_t)INT32_MAX ? (int64_t)INT32_MAX : a;
        a = a < (int64_t)INT32_MIN ? (int64_t)INT32_MIN : a;
        v[i] = (int32_t)a;
      }
    }
#pragma unroll
    for (int i = 0; i < NI; ++i) {
      const int ow = owb + i;
      if (ow < P.OW) {
        int32_t o = v[i];
        if (resid) o = add_sat(o, __ldg(P.residual + rowbase + ow));
        if (relu) o = max(o, 0);
        amax_local = max(amax_local, uabs(o));
        v[i] = o;
      }
    }
    if (NI % 4 == 0 && (P.OW & 3) == 0 && owb + NI <= P.OW) {
#pragma unroll
      for (int q = 0; q < NI / 4; ++q)
        *reinterpret_cast<int4*>(P.y + rowbase + owb + 4 * q) =
            make_int4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    } else {
#pragma unroll
      for (int i = 0; i < NI; ++i)
        if (owb + i < P.OW) P.y[rowbase + owb + i] = v[i];
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
      if (hi != 0ull || lo > ~0ull - 32767ull) {
        unsafe = true;
      } else {
        unsafe = (((lo + 32767ull) >> 15) + nnz + b) > (unsigned long long)INT32_MAX;
      }
    }
  }
  return !__syncthreads_or(unsafe);
}

template <int SIG, int S>
__global__ void __launch_bounds__(kMaxThreads, 3) conv_direct_kernel(const GemmParams P, const DirectGeom G) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int tiles_w = (P.OW + 8 * G.GW - 1) / (8 * G.GW);
  const int tiles_h = (P.OH + G.TH - 1) / G.TH;
  int bx = blockIdx.x;
  const int tw = bx % tiles_w;
  bx /= tiles_w;
  const int th = bx % tiles_h;
  const int n_img = bx / tiles_h;
  const int64_t col0 = (int64_t)blockIdx.y * NT;
  const int oh0 = th * G.TH, ow0 = tw * 8 * G.GW;

  uint32_t amax_local = 0;
  if (tile_int32_exact(P, col0)) {
    run_direct<SIG, S, 0, TM, uint32_t>(P, G, smem_raw, n_img, oh0, ow0, col0, amax_local);
  } else {
    run_direct<SIG, S, 0, TM / 2, int64_t>(P, G, smem_raw, n_img, oh0, ow0, col0, amax_local);
    run_direct<SIG, S, TM / 2, TM / 2, int64_t>(P, G, smem_raw, n_img, oh0, ow0, col0, amax_local);
  }
  if (P.amax_out != nullptr) {
    amax_local = __reduce_max_sync(0xffffffffu, amax_local);
    if ((threadIdx.x & 31) == 0 && amax_local) atomicMax(P.amax_out, amax_local);
  }
}

// Tile choice: 8-column groups to cover the output row (at most 8), then rows
// so that the CTA has at most 256 threads.
DirectGeom choose_geom(const GemmParams& p) {
  DirectGeom G;
  G.GW = (p.OW + 7) / 8;
  if (G.GW > 8) {
    // split wide rows into equal pieces of at most 8 groups
    const int pieces = (G.GW + 7) / 8;
    G.GW = (G.GW + pieces - 1) / pieces;
  }
  const int max_rows = kMaxThreads / (G.GW * CG);
  G.TH = max_rows < 1 ? 1 : max_rows;
  if (G.TH > p.OH) G.TH = p.OH;
  // whole warps only: GW * TH even
  if ((G.GW * G.TH) & 1) G.TH = (G.TH + 1 <= max_rows) ? G.TH + 1 : G.TH - 1;
  if (G.TH < 1) G.TH = 1;
  const int RS = p.R * p.S;
  int cc = RS == 1 ? 32 : (RS <= 9 ? 4 : (RS <= 25 ? 2 : 1));
  if (cc > p.C) cc = p.C;
  G.CC = cc;
  G.HR = (G.TH - 1) * p.sh + p.R;
  const int WS = 7 * p.sw + p.S;
  const int WV4 = (WS + 3) / 4 * 4;
  const int hwd = (8 * G.GW - 1) * p.sw + p.S;
  int hwp = (G.GW - 1) * 8 * p.sw + WV4;
  if (hwp < hwd) hwp = hwd;
  G.HWP = (hwp + 3) / 4 * 4;
  G.taps = G.CC * RS;
  G.n_stages = (p.C + G.CC - 1) / G.CC;
  G.halo_words = G.CC * G.HR * G.HWP;
  G.code_words = G.taps * NT;
  G.threads = G.TH * G.GW * CG;
  return G;
}

template <int SIG, int S>
cudaError_t launch_direct(const GemmParams& p, const DirectGeom G, cudaStream_t st) {
  const size_t smem = (size_t)2 * (G.halo_words + 2 * G.code_words) * sizeof(int32_t);
  cudaError_t e = cudaFuncSetAttribute(conv_direct_kernel<SIG, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const int tiles_w = (p.OW + 8 * G.GW - 1) / (8 * G.GW);
  const int tiles_h = (p.OH + G.TH - 1) / G.TH;
  const int64_t nb = (int64_t)tiles_w * tiles_h * (p.rows / ((int64_t)p.OH * p.OW));
  dim3 grid((unsigned)nb, (unsigned)((p.cols + NT - 1) / NT));
  conv_direct_kernel<SIG, S><<<grid, G.threads, smem, st>>>(p, G);
  return cudaGetLastError();
}

}  // namespace

bool conv_direct_supported(const GemmParams& p) {
  if (p.sh != p.sw) return false;
  if (!(p.sh == 1 || p.sh == 2)) return false;
  if (!(p.S == 1 || p.S == 3 || p.S == 7)) return false;
  if (p.R > 7) return false;
  const DirectGeom G = choose_geom(p);
  const size_t smem = (size_t)2 * (G.halo_words + 2 * G.code_words) * sizeof(int32_t);
  return smem <= 200 * 1024 && G.threads >= NT && (G.threads % 32) == 0 &&
         (p.rows / ((int64_t)p.OH * p.OW)) < (int64_t)1 << 24;
}

cudaError_t launch_conv2d_direct(const GemmParams& p, cudaStream_t st) {
  const DirectGeom G = choose_geom(p);
  if (p.sh == 1) {
    if (p.S == 1) return launch_direct<1, 1>(p, G, st);
    if (p.S == 3) return launch_direct<1, 3>(p, G, st);
    return launch_direct<1, 7>(p, G, st);
  }
  if (p.S == 1) return launch_direct<2, 1>(p, G, st);
  if (p.S == 3) return launch_direct<2, 3>(p, G, st);
  return launch_direct<2, 7>(p, G, st);
}

}  // namespace ds
