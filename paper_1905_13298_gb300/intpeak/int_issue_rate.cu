// Integer issue-rate microbenchmark for the roofline denominator of the
// shift kernels (built as its own small library, not part of the C ABI).
// A DeepShift term (Eq. 1-2: a shift and a sign flip, the multiply of Fig. 1a
// replaced) is SHF + IMAD here, so kind 2 measures the rate a term loop can
// reach.
//
// Each kernel runs a register-resident loop of one instruction mix with
// enough independent chains to hide latency over a grid of CTAs, and records
// per CTA its SM and its first and last clock64() (one counter per SM).
// ops/clk/SM = thread instructions of the mix executed by the CTAs of one SM
// / (last end - first start on that SM), so a mix whose registers allow fewer
// resident CTAs (which then run one after the other) is not over-counted.
//   kind 0: SHF only        (shr.s32, ALU pipe)
//   kind 1: IMAD only       (mad.lo.s32, FMA pipe)
//   kind 2: SHF + IMAD      (the shift-GEMM inner loop: t = x >> s; acc += g * t)
//   kind 3: IADD3 only      (add.s32 chains)
//   kind 4: LOP3 only       (xor/and chains)
//   kind 5: IMAD.HI only    (mad.hi.s32: high word of x * m plus acc)
//   kind 6: IADD3 pairs     (acc = acc + a + b, three-input adds)
//   kind 7: SWAR pair       (two 16-bit activations per register, Sec. 5.2.1's narrow format: one shift
//                            of both lanes, one LOP3 (t & m) ^ c that clears the high lane's bits shifted
//                            into the low lane and flips the lanes' sign bits for the sign extension,
//                            whose constant is folded into a per-column correction, and one IMAD by the
//                            sign: 3 instructions per 2 terms)
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

template <int KIND>
__global__ void __launch_bounds__(256) mix_kernel(const int* __restrict__ seed, int iters, int* out,
                                                  long long* cycles, int* smid) {
  int x[8], s[8], g[8], m[8], c[8], acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    x[i] = seed[(threadIdx.x + i) & 63];
    s[i] = seed[64 + i] & 15;
    g[i] = seed[72 + i];
    m[i] = seed[(64 + 3 * i) & 79] | 0x0000ffff;
    c[i] = seed[(72 + 5 * i) & 79] & 0x80008000;
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = i ^ j;
  }
  __syncthreads();
  const long long t0 = clock64();
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (KIND == 0) {
          asm volatile("shr.s32 %0, %0, %1;" : "+r"(acc[i][j]) : "r"(s[j]));
        } else if (KIND == 1) {
          asm volatile("mad.lo.s32 %0, %0, %1, %2;" : "+r"(acc[i][j]) : "r"(g[j]), "r"(x[i]));
        } else if (KIND == 2) {
          int t;
          asm volatile("shr.s32 %0, %1, %2;" : "=r"(t) : "r"(x[i]), "r"(s[j]));
          asm volatile("mad.lo.s32 %0, %1, %2, %0;" : "+r"(acc[i][j]) : "r"(g[j]), "r"(t));
        } else if (KIND == 3) {
          asm volatile("add.s32 %0, %0, %1;" : "+r"(acc[i][j]) : "r"(x[i]));
        } else if (KIND == 5) {
          asm volatile("mad.hi.s32 %0, %1, %2, %0;" : "+r"(acc[i][j]) : "r"(x[i]), "r"(g[j]));
        } else if (KIND == 7) {
          int t;
          asm volatile("shr.s32 %0, %1, %2;" : "=r"(t) : "r"(x[i]), "r"(s[j]));
          asm volatile("lop3.b32 %0, %0, %1, %2, 0x6A;" : "+r"(t) : "r"(m[j]), "r"(c[j]));
          asm volatile("mad.lo.s32 %0, %1, %2, %0;" : "+r"(acc[i][j]) : "r"(g[j]), "r"(t));
        } else if (KIND == 6) {
          asm volatile("{\n\t.reg .s32 t;\n\tadd.s32 t, %1, %2;\n\tadd.s32 %0, %0, t;\n\t}" : "+r"(acc[i][j]) : "r"(x[i]), "r"(g[j]));
        } else {
          asm volatile("xor.b32 %0, %0, %1;" : "+r"(acc[i][j]) : "r"(g[j]));
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] += acc[i][i];
  }
  const long long t1 = clock64();
  int r = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) r ^= acc[i][j];
  out[blockIdx.x * blockDim.x + threadIdx.x] = r;
  if (threadIdx.x == 0) {
    unsigned sm;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
    cycles[2 * blockIdx.x] = t0;
    cycles[2 * blockIdx.x + 1] = t1;
    smid[blockIdx.x] = (int)sm;
  }
}

}  // namespace

// Runs one mix; writes per CTA its (start, end) clock64 pair and SM id, and
// the kernel time (ms).  out must hold blocks*threads ints, cycles 2*blocks
// long longs, smid `blocks` ints, seed 80 ints.
extern "C" int ds_probe_int_mix(int kind, int blocks, int threads, int iters, const int* seed, int* out,
                                long long* cycles, int* smid, float* ms) {
  cudaEvent_t a, b;
  cudaEventCreate(&a);
  cudaEventCreate(&b);
  cudaEventRecord(a);
  switch (kind) {
    case 0: mix_kernel<0><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 1: mix_kernel<1><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 2: mix_kernel<2><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 3: mix_kernel<3><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 5: mix_kernel<5><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 6: mix_kernel<6><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    case 7: mix_kernel<7><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
    default: mix_kernel<4><<<blocks, threads>>>(seed, iters, out, cycles, smid); break;
  }
  cudaEventRecord(b);
  cudaError_t e = cudaEventSynchronize(b);
  cudaEventElapsedTime(ms, a, b);
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  return e == cudaSuccess ? (int)cudaGetLastError() : (int)e;
}
