// Weight-specialised ConvShift (DeepShift Eq. 1-3 on the Sec. 4 fixed point;
// the paper names run-time specialisation of its kernels as future work,
// Sec. 6.1).
//
// For a layer whose codes are few enough to live in the instruction stream,
// the library writes a CUDA kernel in which every weight's shift amount and
// sign are immediates and the zero weights are absent, compiles it at run
// time with NVRTC (opened with dlopen on first use, so the library does not
// depend on it otherwise) into a cubin for the device's architecture, and
// loads it with the runtime's library API.  Per term the kernel issues one
// shift by an immediate and one add or subtract (a weight with p = 0 needs
// no shift), with no shared-memory code loads and no code staging.
//
// Kernel shape: a CTA computes TH output rows x GW groups of TM = 7 pixels of
// one image for CPT output channels, every thread the same channels (so that
// a CTA, and the CTAs launched next to it, run one channel group's code and
// the instruction working set stays one group's); CPT is the largest of 4, 2,
// 1 with at most 2048 terms per thread and group.  The CTA stages the input
// window of every pixel group for all C channels once (C is small: the first
// layers of a network), then runs its group's straight-line code: per (c, r)
// one window load from shared memory, reused by the S taps and CPT channels.
// Accumulator width as everywhere in the library: the per-channel constants
// A[n] and nnz[n] of the bound are immediates, max|x| and the bias are read
// at run time, and a CTA whose channels the bound does not cover runs the
// same code on 64-bit accumulators and saturates.
#include <dlfcn.h>
#include <nvrtc.h>  // types only: the functions are looked up in the library at run time

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <mutex>
#include <string>
#include <vector>

#include "ds_common.cuh"

struct ds_specialized {
  cudaLibrary_t lib;
  cudaKernel_t kern;
  int K, C, R, S, stride, pad;
  int TH, GW, TM, CPT, groups;
  size_t smem;
};

namespace ds {
namespace {

constexpr int kTM = 7;
constexpr int kGW = 8;
constexpr int kMaxTermsPerThread = 2048;
constexpr size_t kMaxSmem = 96 * 1024;

struct Nvrtc {
  decltype(&nvrtcCreateProgram) create = nullptr;
  decltype(&nvrtcCompileProgram) compile = nullptr;
  decltype(&nvrtcGetProgramLogSize) log_size = nullptr;
  decltype(&nvrtcGetProgramLog) log = nullptr;
  decltype(&nvrtcGetCUBINSize) cubin_size = nullptr;
  decltype(&nvrtcGetCUBIN) cubin = nullptr;
  decltype(&nvrtcDestroyProgram) destroy = nullptr;
  bool ok = false;
};

// NVRTC, opened once per process.
const Nvrtc& nvrtc() {
  static const Nvrtc n = [] {
    Nvrtc r;
    void* h = nullptr;
    for (const char* name : {"libnvrtc.so.13", "libnvrtc.so", "/usr/local/cuda/lib64/libnvrtc.so.13"}) {
      h = dlopen(name, RTLD_NOW | RTLD_LOCAL);
      if (h) break;
    }
    if (!h) return r;
    r.create = reinterpret_cast<decltype(r.create)>(dlsym(h, "nvrtcCreateProgram"));
    r.compile = reinterpret_cast<decltype(r.compile)>(dlsym(h, "nvrtcCompileProgram"));
    r.log_size = reinterpret_cast<decltype(r.log_size)>(dlsym(h, "nvrtcGetProgramLogSize"));
    r.log = reinterpret_cast<decltype(r.log)>(dlsym(h, "nvrtcGetProgramLog"));
    r.cubin_size = reinterpret_cast<decltype(r.cubin_size)>(dlsym(h, "nvrtcGetCUBINSize"));
    r.cubin = reinterpret_cast<decltype(r.cubin)>(dlsym(h, "nvrtcGetCUBIN"));
    r.destroy = reinterpret_cast<decltype(r.destroy)>(dlsym(h, "nvrtcDestroyProgram"));
    r.ok = r.create && r.compile && r.log_size && r.log && r.cubin_size && r.cubin && r.destroy;
    return r;
  }();
  return n;
}

void append(std::string& s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  const int n = vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (n > 0) s.append(buf, std::min<size_t>((size_t)n, sizeof(buf) - 1));
}

// The kernel source of one layer.  s, p: host codes [K][C][R][S].
std::string kernel_source(const int8_t* s, const int8_t* p, const ds_specialized& h, int WS, int WV, int WSP,
                          int HR) {
  std::string src;
  src.reserve(1 << 20);
  append(src,
         "typedef unsigned int u32; typedef unsigned long long u64; typedef long long i64;\n"
         "#define K_ %d\n#define C_ %d\n#define R_ %d\n#define S_ %d\n#define STR %d\n#define PAD %d\n"
         "#define TM %d\n#define GW %d\n#define TH %d\n#define CPT %d\n#define HR %d\n#define WS %d\n"
         "#define WV %d\n#define WSP %d\n#define NTHREADS %d\n",
         h.K, h.C, h.R, h.S, h.stride, h.pad, h.TM, h.GW, h.TH, h.CPT, HR, WS, WV, WSP, h.TH * h.GW);
  src +=
      // whether 32-bit accumulation is exact for a column: ceil(amax A / 2^15) + nnz + |b| <= 2^31 - 1
      "__device__ __forceinline__ bool fits(u64 amax, u64 A, u64 nnz, const int* bias, int col) {\n"
      "  const u64 b = bias ? (u64)(bias[col] < 0 ? 0u - (u32)bias[col] : (u32)bias[col]) : 0ull;\n"
      "  const u64 hi = __umul64hi(amax, A), lo = amax * A;\n"
      "  if (hi != 0ull || lo > ~0ull - 32767ull) return false;\n"
      "  return ((lo + 32767ull) >> 15) + nnz + b <= 2147483647ull;\n}\n"
      "__device__ __forceinline__ int add_sat(int a, int b) { int r; asm(\"add.sat.s32 %0, %1, %2;\" : \"=r\"(r) : "
      "\"r\"(a), \"r\"(b)); return r; }\n"
      // window of kernel row r of channel c: WV 16-byte loads from the thread's slot
      "#define LOADW(c, r) { const int4* wp = (const int4*)(hb + ((c) * HR + (r)) * GW * WSP); _Pragma(\"unroll\") "
      "for (int v = 0; v < WV; ++v) { const int4 q = wp[v]; w[4*v] = q.x; w[4*v+1] = q.y; w[4*v+2] = q.z; "
      "w[4*v+3] = q.w; } }\n"
      // one weight (tap s of channel j of the group): + or - (x >> k) on the TM pixels
      "#define TP(j, s, k) { _Pragma(\"unroll\") for (int i = 0; i < TM; ++i) a[j][i] += (acc_t)(w[i * STR + (s)] >> "
      "(k)); }\n"
      "#define TN(j, s, k) { _Pragma(\"unroll\") for (int i = 0; i < TM; ++i) a[j][i] -= (acc_t)(w[i * STR + (s)] >> "
      "(k)); }\n";

  // the body of one channel group: the straight-line terms; BODY_<g>(T)
  for (int grp = 0; grp < h.groups; ++grp) {
    append(src, "#define BODY_%d { ", grp);
    for (int c = 0; c < h.C; ++c)
      for (int r = 0; r < h.R; ++r) {
        std::string terms;
        for (int q = 0; q < h.S; ++q)
          for (int j = 0; j < h.CPT; ++j) {
            const int col = grp * h.CPT + j;
            if (col >= h.K) continue;
            const int64_t idx = (((int64_t)col * h.C + c) * h.R + r) * h.S + q;
            const int sv = s[idx], pv = p[idx];
            if (sv == 0) continue;  // a zero weight is absent from the code
            append(terms, sv > 0 ? "TP(%d,%d,%d)" : "TN(%d,%d,%d)", j, q, -pv);
          }
        if (!terms.empty()) {
          append(src, "LOADW(%d,%d) ", c, r);
          src += terms;
          src += " ";
        }
      }
    src += "}\n";
  }

  // the terms of the CTA's channel group on accumulators of type acc_t, then the epilogue: bias,
  // saturation (64-bit), residual, ReLU, max|y|, store
  src +=
      "template <typename acc_t>\n"
      "__device__ __forceinline__ void run(const int* hb, int grp, int* y, const int* bias, const int* residual,\n"
      "                                    i64 n, int oh, int owb, int OH, int OW, bool relu, bool resid,\n"
      "                                    u32& amax_l) {\n"
      "  acc_t a[CPT][TM];\n"
      "  _Pragma(\"unroll\") for (int j = 0; j < CPT; ++j) _Pragma(\"unroll\") for (int i = 0; i < TM; ++i) "
      "a[j][i] = 0;\n"
      "  int w[WV * 4];\n"
      "  switch (grp) {\n";
  for (int grp = 0; grp < h.groups; ++grp) append(src, "    case %d: BODY_%d break;\n", grp, grp);
  src +=
      "  }\n"
      "  if (oh >= OH) return;\n"
      "  _Pragma(\"unroll\") for (int j = 0; j < CPT; ++j) {\n"
      "    const int col = grp * CPT + j;\n"
      "    if (col >= K_) break;\n"
      "    const i64 b = bias ? (i64)bias[col] : 0;\n"
      "    int* yr = y + ((n * K_ + col) * OH + oh) * (i64)OW;\n"
      "    const int* rr = resid ? residual + ((n * K_ + col) * OH + oh) * (i64)OW : 0;\n"
      "    _Pragma(\"unroll\") for (int i = 0; i < TM; ++i) {\n"
      "      const int ow = owb + i;\n"
      "      if (ow >= OW) break;\n"
      "      int o;\n"
      "      if (sizeof(acc_t) == 4) {\n"
      "        o = (int)((u32)a[j][i] + (u32)b);\n"
      "      } else {\n"
      "        i64 v = (i64)a[j][i] + b;\n"
      "        v = v > 2147483647ll ? 2147483647ll : (v < -2147483648ll ? -2147483648ll : v);\n"
      "        o = (int)v;\n"
      "      }\n"
      "      if (resid) o = add_sat(o, rr[ow]);\n"
      "      if (relu) o = o > 0 ? o : 0;\n"
      "      const u32 m = o < 0 ? 0u - (u32)o : (u32)o;\n"
      "      amax_l = m > amax_l ? m : amax_l;\n"
      "      yr[ow] = o;\n"
      "    }\n"
      "  }\n"
      "}\n";
  src +=
      "extern \"C\" __global__ void __launch_bounds__(NTHREADS, 4) ds_shift_conv_specialized(\n"
      "    const int* __restrict__ x, int* __restrict__ y, const int* __restrict__ bias,\n"
      "    const int* __restrict__ residual, const u32* __restrict__ amax_in, u32* __restrict__ amax_out,\n"
      "    int H, int W, int OH, int OW, u32 flags, int tiles_w, int tiles_h) {\n"
      "  extern __shared__ __align__(16) int halo[];\n"
      "  const int t = threadIdx.x;\n"
      "  const int g = t % GW, oh_l = t / GW;\n"
      "  const int tw = blockIdx.x % tiles_w;\n"
      "  const int rest = blockIdx.x / tiles_w;\n"
      "  const int th = rest % tiles_h;\n"
      "  const i64 n = rest / tiles_h;\n"
      "  const int oh0 = th * TH, ow0 = tw * TM * GW;\n"
      "  const int grp = blockIdx.y;\n"
      // the input windows of all C channels: slot (c, hr, gg) holds input row oh0*STR - PAD + hr, columns
      // (ow0 + gg*TM)*STR - PAD + [0, WS); zero outside the image
      "  const i64 HW = (i64)H * W;\n"
      "  for (int sl = t; sl < C_ * HR * GW; sl += NTHREADS) {\n"
      "    const int gg = sl % GW, row = sl / GW, hr = row % HR, c = row / HR;\n"
      "    const int ih = oh0 * STR - PAD + hr;\n"
      "    const int iws = (ow0 + gg * TM) * STR - PAD;\n"
      "    const bool rok = (unsigned)ih < (unsigned)H;\n"
      "    const int* src = x + (n * C_ + c) * HW + (i64)(rok ? ih : 0) * W;\n"
      "    const u32 d0 = (u32)__cvta_generic_to_shared(halo + sl * WSP);\n"
      "    _Pragma(\"unroll\") for (int i = 0; i < WS; ++i) {\n"
      "      const bool ok = rok && (unsigned)(iws + i) < (unsigned)W;\n"
      "      asm volatile(\"cp.async.ca.shared.global [%0], [%1], 4, %2;\" :: \"r\"(d0 + 4u * i),\n"
      "                   \"l\"(ok ? (const void*)(src + iws + i) : (const void*)x), \"r\"(ok ? 4 : 0));\n"
      "    }\n"
      "  }\n"
      "  asm volatile(\"cp.async.commit_group;\");\n"
      // the bound, per channel of the group (A, nnz immediates; max|x| and bias at run time)
      "  bool exact = amax_in != 0 && !(flags & 16u);\n"
      "  const u64 amax = amax_in ? (u64)*amax_in : 0ull;\n"
      "  switch (grp) {\n";
  for (int grp = 0; grp < h.groups; ++grp) {
    append(src, "    case %d:", grp);
    for (int j = 0; j < h.CPT; ++j) {
      const int col = grp * h.CPT + j;
      if (col >= h.K) continue;
      unsigned long long A = 0;
      unsigned nnz = 0;
      for (int64_t e = 0; e < (int64_t)h.C * h.R * h.S; ++e) {
        const int64_t idx = (int64_t)col * h.C * h.R * h.S + e;
        if (s[idx] != 0) {
          A += 1ull << (15 + p[idx]);
          ++nnz;
        }
      }
      append(src, " exact = exact && fits(amax, %lluull, %uull, bias, %d);", A, nnz, col);
    }
    src += " break;\n";
  }
  src +=
      "  }\n"
      "  asm volatile(\"cp.async.wait_group 0;\" ::: \"memory\");\n"
      "  __syncthreads();\n"
      "  const int* hb = halo + (oh_l * STR * GW + g) * WSP;\n"
      "  const bool relu = (flags & 1u) != 0, resid = (flags & 8u) != 0 && residual != 0;\n"
      "  u32 amax_l = 0;\n"
      "  if (exact) run<u32>(hb, grp, y, bias, residual, n, oh0 + oh_l, ow0 + g * TM, OH, OW, relu, resid, amax_l);\n"
      "  else run<i64>(hb, grp, y, bias, residual, n, oh0 + oh_l, ow0 + g * TM, OH, OW, relu, resid, amax_l);\n"
      "  if (amax_out) {\n"
      "    amax_l = __reduce_max_sync(0xffffffffu, amax_l);\n"
      "    if ((t & 31) == 0 && amax_l) atomicMax(amax_out, amax_l);\n"
      "  }\n"
      "}\n";
  return src;
}

}  // namespace

ds_status specialize_conv(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride, int pad,
                          ds_specialized** out) {
  *out = nullptr;
  const Nvrtc& rt = nvrtc();
  if (!rt.ok) return fail(DS_ERR_UNSUPPORTED, "weight specialisation needs NVRTC (libnvrtc.so), not found");
  int dev = 0, major = 0, minor = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (e != cudaSuccess) return cuda_check(e, "device query");

  ds_specialized h{};
  h.K = K;
  h.C = C;
  h.R = R;
  h.S = S;
  h.stride = stride;
  h.pad = pad;
  h.TM = kTM;
  h.GW = kGW;
  const int taps = C * R * S;
  h.CPT = 1;
  for (int cpt : {4, 2}) {
    if (taps * kTM * cpt <= kMaxTermsPerThread && cpt <= K) {
      h.CPT = cpt;
      break;
    }
  }
  h.groups = (K + h.CPT - 1) / h.CPT;
  const int WS = (kTM - 1) * stride + S;
  const int WV = (WS + 3) / 4;
  const int WSP = WV * 4 + (WV % 2 == 0 ? 4 : 0);
  int HR = 0;
  for (int th : {16, 8, 4}) {
    h.TH = th;
    HR = (th - 1) * stride + R;
    h.smem = (size_t)C * HR * kGW * WSP * sizeof(int32_t);
    if (h.smem <= kMaxSmem) break;
  }
  if (h.smem > kMaxSmem)
    return fail(DS_ERR_UNSUPPORTED, "the input windows of %d channels need %zu bytes of shared memory", C, h.smem);

  const std::string src = kernel_source(s, p, h, WS, WV, WSP, HR);
  nvrtcProgram prog;
  if (rt.create(&prog, src.c_str(), "ds_specialized.cu", 0, nullptr, nullptr) != NVRTC_SUCCESS)
    return fail(DS_ERR_UNSUPPORTED, "NVRTC could not create the program");
  char arch[64];
  snprintf(arch, sizeof(arch), "-arch=sm_%d%d%s", major, minor, major >= 9 ? "a" : "");
  const char* opts[] = {arch, "-std=c++17", "-default-device"};
  const nvrtcResult cr = rt.compile(prog, 3, opts);
  if (cr != NVRTC_SUCCESS) {
    size_t n = 0;
    rt.log_size(prog, &n);
    std::string log(n, '\0');
    if (n) rt.log(prog, &log[0]);
    rt.destroy(&prog);
    return fail(DS_ERR_UNSUPPORTED, "NVRTC compile failed: %.300s", log.c_str());
  }
  size_t nbin = 0;
  rt.cubin_size(prog, &nbin);
  std::vector<char> bin(nbin);
  if (nbin == 0 || rt.cubin(prog, bin.data()) != NVRTC_SUCCESS) {
    rt.destroy(&prog);
    return fail(DS_ERR_UNSUPPORTED, "NVRTC produced no cubin");
  }
  rt.destroy(&prog);
  e = cudaLibraryLoadData(&h.lib, bin.data(), nullptr, nullptr, 0, nullptr, nullptr, 0);
  if (e != cudaSuccess) return cuda_check(e, "loading the specialised kernel");
  e = cudaLibraryGetKernel(&h.kern, h.lib, "ds_shift_conv_specialized");
  if (e == cudaSuccess && h.smem > 48 * 1024)
    e = cudaKernelSetAttributeForDevice(h.kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)h.smem, dev);
  if (e != cudaSuccess) {
    (void)cudaLibraryUnload(h.lib);
    return cuda_check(e, "the specialised kernel");
  }
  ds_specialized* r = new (std::nothrow) ds_specialized(h);
  if (!r) {
    (void)cudaLibraryUnload(h.lib);
    return fail(DS_ERR_UNSUPPORTED, "host allocation of the specialised layer failed");
  }
  *out = r;
  return DS_OK;
}

cudaError_t launch_specialized(const ds_specialized* h, const int32_t* x, const int32_t* bias,
                               const int32_t* residual, int32_t* y, int N, int H, int W, int OH, int OW,
                               uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out, cudaStream_t st) {
  const int tiles_w = (OW + h->TM * h->GW - 1) / (h->TM * h->GW);
  const int tiles_h = (OH + h->TH - 1) / h->TH;
  const int64_t nx = (int64_t)N * tiles_h * tiles_w;
  if (nx > INT32_MAX || h->groups > 65535) return cudaErrorInvalidConfiguration;
  void* args[] = {(void*)&x, (void*)&y, (void*)&bias, (void*)&residual, (void*)&amax_in, (void*)&amax_out,
                  (void*)&H, (void*)&W, (void*)&OH, (void*)&OW, (void*)&flags, (void*)&tiles_w, (void*)&tiles_h};
  return cudaLaunchKernel((const void*)h->kern, dim3((unsigned)nx, (unsigned)h->groups, 1),
                          dim3((unsigned)(h->TH * h->GW), 1, 1), args, h->smem, st);
}

void specialized_dims(const ds_specialized* h, int* K, int* C, int* R, int* S, int* stride, int* pad) {
  *K = h->K;
  *C = h->C;
  *R = h->R;
  *S = h->S;
  *stride = h->stride;
  *pad = h->pad;
}

void destroy_specialized(ds_specialized* h) {
  if (!h) return;
  (void)cudaLibraryUnload(h->lib);
  delete h;
}

}  // namespace ds
