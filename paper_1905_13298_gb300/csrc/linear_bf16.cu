// Float variant of LinearShift on the 5th-generation tensor cores (sm_103a).
//
//   y[m][n] = ReLU?( bias[n] + sum_k x[m][k] * W[n][k] ),   W = flip(2^P, S)   (Eq. 3)
//
// x is bf16, W = s * 2^p is exact in bf16 (sign bit, exponent 127 + p, zero
// mantissa; s = 0 gives +0), so every product is exact and only the fp32
// accumulation rounds.  This is a dense contraction, so it runs as a GEMM.
// Persistent: one CTA per SM walks the 128 x 256 output tiles t = blockIdx.x,
// blockIdx.x + gridDim.x, ... in grouped order (tile_of): groups of G row
// tiles, n fastest inside a group, with G x (column tiles) about one wave, so
// the tiles in flight share their x rows and W rows in L2.  6 warps:
//   warp 0     one elected thread issues TMA loads (128B-swizzled K-major
//              tiles of 64 bf16) into a 4-stage shared-memory ring that runs
//              on across tiles,
//   warp 1     allocates 512 TMEM columns: two 256-column fp32 accumulators.
//              One thread issues tcgen05.mma (kind::f16, M=128, N=256, K=16)
//              for tile i into accumulator i % 2, frees each ring slot with
//              tcgen05.commit and commits the tile to tfull[i % 2],
//   warps 2-5  wait for tfull, read the accumulator with tcgen05.ld (one TMEM
//              lane quarter per warp), release it (tempty) and add the bias,
//              apply ReLU and store fp32 rows, while the MMAs of the next
//              tile run into the other accumulator.
// mbarriers: full[s] (TMA bytes landed), empty[s] (MMAs done reading slot s),
// tfull[b] (tile's MMAs done), tempty[b] (accumulator b read out), done (all
// MMAs of the CTA finished, waited for before TMEM is freed).  Every wait is
// bounded by a clock deadline; on expiry the kernel records a fault flag,
// stops issuing work, waits (bounded) for issued work and frees its TMEM.
#include <cuda.h>

#include <atomic>
#include <cudaTypedefs.h>

#include "ds_common.cuh"

namespace ds {

__device__ int g_bf16_fault;  // set when a bounded wait of the bf16 kernel gives up

namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;  // 16 KB
constexpr int B_BYTES = BN * BK * 2;  // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int ACC_BUFS = 2;
constexpr int TMEM_COLS = ACC_BUFS * BN;  // 512: the whole tensor memory of an SM
constexpr int kThreads = 192;
constexpr int kEpiWarps = 4;
constexpr long long kTimeoutCycles = 4000000000LL;  // about 2 s at 2 GHz
// the wait limit of the next launches (a diagnostic can shorten it to make the waits run out)
std::atomic<long long> g_wait_cycles{kTimeoutCycles};

struct Bf16Params {
  float* y;
  const float* bias;
  int64_t M, N, K;
  uint32_t flags;
  long long wait_cycles;  // limit of a bounded wait before the launch gives up (the fault flag)
};

struct __align__(8) Barriers {
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t tfull[ACC_BUFS];
  uint64_t tempty[ACC_BUFS];
  uint64_t done;
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity; false when the CTA
// aborted or the deadline passed (then the fault flag and abort are set).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort, long long limit) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort) return false;
    if (clock64() - t0 > limit) {
      *abort = 1;
      atomicExch(&g_bf16_fault, 1);
      return false;
    }
  }
  return true;
}
// Bounded wait that ignores the abort flag (draining work already issued);
// always the full limit, so that issued copies and MMAs land before the CTA
// frees its tensor memory or exits.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity) && clock64() - t0 < kTimeoutCycles) {
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::
          "r"(smem_u32(dst)),
      "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile with 128-byte swizzle:
// rows of 128 bytes, 8-row groups 1024 bytes apart (tile base 1024-aligned).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
  uint64_t d = (uint64_t)((addr >> 4) & 0x3FFFu);  // start address
  d |= (uint64_t)1 << 16;                          // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;                // stride byte offset
  d |= (uint64_t)1 << 46;                          // descriptor version of this architecture
  d |= (uint64_t)2 << 61;                          // 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16 with bf16 A and B (K-major), fp32 D, M = 128, N = 256.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// Tile t of the grouped order: rows [m0, m0 + BM), columns [n0, n0 + BN).
__device__ __forceinline__ void tile_of(int64_t t, int64_t tiles_m, int64_t tiles_n, int64_t G, int& m0, int& n0) {
  const int64_t per_group = G * tiles_n;
  const int64_t first_m = (t / per_group) * G;
  const int64_t gsize = tiles_m - first_m < G ? tiles_m - first_m : G;
  const int64_t r = t - (t / per_group) * per_group;
  m0 = (int)((first_m + r % gsize) * BM);
  n0 = (int)((r / gsize) * BN);
}

__global__ void __launch_bounds__(kThreads, 1)
    linear_bf16_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_w,
                       const Bf16Params P) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte aligned stage buffers (the swizzle pattern repeats every 1024 bytes)
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  Barriers* bars = reinterpret_cast<Barriers*>(smem + STAGES * STAGE_BYTES);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t tiles_m = (P.M + BM - 1) / BM;
  const int64_t tiles_n = (P.N + BN - 1) / BN;
  const int64_t ntiles = tiles_m * tiles_n;
  // rows tiles per group: about one wave of CTAs per group
  int64_t G = (gridDim.x + tiles_n - 1) / tiles_n;
  G = G < 1 ? 1 : (G > tiles_m ? tiles_m : G);
  const int nk = (int)((P.K + BK - 1) / BK);
  volatile int* abort = &bars->abort;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);
    }
    for (int b = 0; b < ACC_BUFS; ++b) {
      mbar_init(&bars->tfull[b], 1);
      mbar_init(&bars->tempty[b], kEpiWarps);
    }
    mbar_init(&bars->done, 1);
    bars->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&bars->tmem_base)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem_base = bars->tmem_base;

  if (warp == 0) {
    if (lane == 0) {  // TMA producer: the ring's slot counter runs on across tiles
      int64_t it = 0;
      bool ok = true;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        int m0, n0;
        tile_of(t, tiles_m, tiles_n, G, m0, n0);
        for (int kt = 0; kt < nk; ++kt, ++it) {
          const int s = (int)(it % STAGES);
          const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
          if (it >= STAGES && !mbar_wait(&bars->empty[s], ph ^ 1u, abort, P.wait_cycles)) {
            ok = false;
            break;
          }
          unsigned char* a = smem + s * STAGE_BYTES;
          mbar_expect_tx(&bars->full[s], STAGE_BYTES);
          tma_load_2d(a, &tmap_x, &bars->full[s], kt * BK, m0);
          tma_load_2d(a + A_BYTES, &tmap_w, &bars->full[s], kt * BK, n0);
        }
      }
      // before leaving, let every issued copy land (bounded): the last
      // STAGES full barriers cover all copies still in flight
      for (int64_t j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
        mbar_drain(&bars->full[j % STAGES], (uint32_t)(j / STAGES) & 1u);
    }
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      int64_t it = 0;
      int64_t i = 0;  // tiles of this CTA so far
      bool ok = true;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++i) {
        const int b = (int)(i & 1);
        // accumulator b is free once the epilogue has read tile i - 2 out of it
        if (i >= ACC_BUFS && !mbar_wait(&bars->tempty[b], (uint32_t)((i / ACC_BUFS) - 1) & 1u, abort, P.wait_cycles)) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t tmem_d = tmem_base + (uint32_t)(b * BN);
        for (int kt = 0; kt < nk; ++kt, ++it) {
          const int s = (int)(it % STAGES);
          const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
          if (!mbar_wait(&bars->full[s], ph, abort, P.wait_cycles)) {
            ok = false;
            break;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t a = smem_u32(smem + s * STAGE_BYTES);
          const uint32_t bb = a + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            umma_bf16(tmem_d, sw128_desc(a + 32 * k), sw128_desc(bb + 32 * k), (kt > 0 || k > 0) ? 1u : 0u);
          umma_commit(&bars->empty[s]);  // slot s is free once these MMAs have read it
        }
        if (ok) umma_commit(&bars->tfull[b]);  // fires when the tile's MMAs have completed
      }
      // every MMA issued by this CTA has completed before TMEM is freed
      umma_commit(&bars->done);
      mbar_drain(&bars->done, 0u);
    }
  } else {
    // epilogue: warps 2..5 own TMEM lane quarters (warp % 4)
    const int q = warp & 3;
    const bool relu = (P.flags & DS_RELU) != 0;
    const bool bias_vec = P.bias != nullptr && (reinterpret_cast<uintptr_t>(P.bias) & 15) == 0;
    int64_t i = 0;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++i) {
      const int b = (int)(i & 1);
      if (!mbar_wait(&bars->tfull[b], (uint32_t)(i / ACC_BUFS) & 1u, abort, P.wait_cycles)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      int tm0, tn0;
      tile_of(t, tiles_m, tiles_n, G, tm0, tn0);
      const int64_t m0 = tm0, n0 = tn0;
      const int64_t row = m0 + 32 * q + lane;
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        const uint32_t taddr = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * BN + c0);
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
            "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
              "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
              "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
              "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
              "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
            : "r"(taddr)
            : "memory");
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (c0 + 32 == BN) {
          // the whole accumulator is in registers: hand it back to the MMA warp
          asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->tempty[b]);
        }
        if (row >= P.M) continue;
        float* yrow = P.y + row * P.N + n0 + c0;
        const int64_t nvalid = P.N - (n0 + c0);
        if (nvalid >= 32 && (P.N & 3) == 0) {
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            float4 bv = make_float4(0.f, 0.f, 0.f, 0.f);
            if (bias_vec) {
              bv = __ldg(reinterpret_cast<const float4*>(P.bias + n0 + c0 + j));
            } else if (P.bias) {
              bv = make_float4(__ldg(P.bias + n0 + c0 + j), __ldg(P.bias + n0 + c0 + j + 1),
                               __ldg(P.bias + n0 + c0 + j + 2), __ldg(P.bias + n0 + c0 + j + 3));
            }
            float4 v;
            v.x = __uint_as_float(r[j]) + bv.x;
            v.y = __uint_as_float(r[j + 1]) + bv.y;
            v.z = __uint_as_float(r[j + 2]) + bv.z;
            v.w = __uint_as_float(r[j + 3]) + bv.w;
            if (relu) {
              v.x = fmaxf(v.x, 0.f);
              v.y = fmaxf(v.y, 0.f);
              v.z = fmaxf(v.z, 0.f);
              v.w = fmaxf(v.w, 0.f);
            }
            *reinterpret_cast<float4*>(yrow + j) = v;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            if (j < nvalid) {
              float v = __uint_as_float(r[j]) + (P.bias ? __ldg(P.bias + n0 + c0 + j) : 0.f);
              yrow[j] = relu ? fmaxf(v, 0.f) : v;
            }
          }
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                 : "memory");
  }
}

// bf16 execution layout of the weights: W[n][k] = bf16(s * 2^p), row stride kpad (a multiple of 8).
__global__ void expand_bf16_kernel(const uint8_t* __restrict__ blob, int64_t n_out, int64_t k_red, int64_t kpad,
                                   uint16_t* __restrict__ out) {
  const BlobLayout L = blob_layout(n_out, k_red);
  const int64_t total = n_out * kpad;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = e / kpad;
    const int64_t k = e - n * kpad;
    uint16_t v = 0;
    if (k < k_red) {
      const int64_t rec = (k >> 5) * n_out + n;
      const uint32_t nib = reinterpret_cast<const uint32_t*>(blob + L.nib + rec * 16)[(k >> 3) & 3];
      const uint2 b = reinterpret_cast<const uint2*>(blob + L.bits + rec * 8)[0];
      const int j = (int)(k & 31);
      const uint32_t sh = (nib >> (4 * (k & 7))) & 15u;  // -p
      if ((b.y >> j) & 1u) v = (uint16_t)((((b.x >> j) & 1u) << 15) | ((127u - sh) << 7));
    }
    out[e] = v;
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  // once per process, thread-safe (function-local static)
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

bool make_map(CUtensorMap* map, const void* ptr, int64_t inner, int64_t outer, int64_t row_stride_elems,
              uint32_t box_outer) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
  cuuint64_t strides[1] = {(cuuint64_t)row_stride_elems * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int64_t bf16_kpad(int64_t k_red) { return (k_red + 7) / 8 * 8; }

cudaError_t launch_expand_bf16(const uint8_t* blob, int64_t n_out, int64_t k_red, uint16_t* out,
                               cudaStream_t st) {
  const int threads = 256;
  const int64_t total = n_out * bf16_kpad(k_red);
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > 65535 * 8) blocks = 65535 * 8;
  expand_bf16_kernel<<<(unsigned)blocks, threads, 0, st>>>(blob, n_out, k_red, bf16_kpad(k_red), out);
  return cudaGetLastError();
}

// x: bf16 [M][K] (K % 8 == 0), w16: bf16 [N][kpad], y: fp32 [M][N].
cudaError_t launch_linear_bf16(const uint16_t* x, const uint16_t* w16, const float* bias, float* y, int64_t M,
                               int64_t K, int64_t N, uint32_t flags, cudaStream_t st) {
  CUtensorMap mx, mw;
  if (!make_map(&mx, x, K, M, K, BM)) return cudaErrorInvalidValue;
  if (!make_map(&mw, w16, K, N, bf16_kpad(K), BN)) return cudaErrorInvalidValue;
  const size_t smem = (size_t)STAGES * STAGE_BYTES + sizeof(Barriers) + 1024;
  // once per process, thread-safe (function-local statics)
  static const cudaError_t attr =
      cudaFuncSetAttribute(linear_bf16_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (attr != cudaSuccess) return attr;
  static const int sms = [] {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
                                                  cudaSuccess) {
      (void)cudaGetLastError();
      return 0;
    }
    return n;
  }();
  if (sms <= 0) return cudaErrorInvalidDevice;
  Bf16Params p{y, bias, M, N, K, flags, g_wait_cycles.load(std::memory_order_relaxed)};
  const int64_t tiles = ((M + BM - 1) / BM) * ((N + BN - 1) / BN);
  const unsigned grid = (unsigned)(tiles < sms ? tiles : sms);  // persistent: one CTA per SM
  linear_bf16_kernel<<<grid, kThreads, smem, st>>>(mx, mw, p);
  return cudaGetLastError();
}

void set_bf16_wait_cycles(long long cycles) {
  g_wait_cycles.store(cycles > 0 ? cycles : kTimeoutCycles, std::memory_order_relaxed);
}

int read_bf16_fault_flag() {
  // read, then clear: the flag covers the float calls since the previous read
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_bf16_fault, sizeof(int)) != cudaSuccess) return -1;
  const int zero = 0;
  if (v != 0 && cudaMemcpyToSymbol(g_bf16_fault, &zero, sizeof(int)) != cudaSuccess) return -1;
  return v;
}

}  // namespace ds
