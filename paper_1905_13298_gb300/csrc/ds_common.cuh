// Shared definitions of the DeepShift CUDA library (sm_103a): the packed code
// layout of Eq. 3's flip(2^P, S) (4 shift bits, a sign plane and a non-zero
// plane per 32-weight chunk), the launch parameters of the shift kernels
// (Eq. 1-3 on Sec. 4's fixed point) and their asynchronous-copy helpers.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "deepshift.h"
#include <nvtx3/nvToolsExt.h>  // header-only: a range costs a pointer test unless a profiler is attached

namespace ds {

// An NVTX range for the time of a scope: the entry points and each layer of a
// chained forward appear by name (and layer index) on a profiler's timeline.
struct NvtxRange {
  explicit NvtxRange(const char* name, int index = -1) {
    nvtxEventAttributes_t a = {};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    if (index >= 0) {
      a.payloadType = NVTX_PAYLOAD_TYPE_INT32;
      a.payload.iValue = index;
    }
    nvtxRangePushEx(&a);
  }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// ---------------------------------------------------------------------------
// Error reporting (thread-local last error, see ds_last_error()).
// ---------------------------------------------------------------------------
void set_error(const char* fmt, ...);
void clear_error();
ds_status fail(ds_status st, const char* fmt, ...);
ds_status cuda_check(cudaError_t e, const char* what);

// ---------------------------------------------------------------------------
// Packed blob geometry (format DS_FORMAT_PLANES6, documented in deepshift.h).
// ---------------------------------------------------------------------------
constexpr int64_t kBlobHeader = 256;
constexpr int kChunk = 32;  // reduction indices per packed chunk

struct BlobLayout {
  int64_t n_chunks, nib, bits, col_a, nnz, total;
};

__host__ __device__ inline BlobLayout blob_layout(int64_t n_out, int64_t k_red) {
  BlobLayout L;
  L.n_chunks = (k_red + kChunk - 1) / kChunk;
  L.nib = kBlobHeader;
  L.bits = L.nib + L.n_chunks * n_out * 16;
  L.col_a = L.bits + L.n_chunks * n_out * 8;
  L.nnz = L.col_a + n_out * 8;
  int64_t end = L.nnz + n_out * 4;
  L.total = (end + 255) / 256 * 256;
  return L;
}

// Header written on the device by the pack kernel.
struct BlobHeader {
  uint32_t magic;
  uint32_t format;
  int64_t n_out;
  int64_t k_red;
  int64_t n_chunks;
  uint32_t invalid_count;
  uint32_t nnz_max;
  unsigned long long a_max;
};
static_assert(sizeof(BlobHeader) == 48, "header layout");

// Division by a runtime constant d >= 1 of numerators 0 <= n < 2^31 as one
// widening multiply and a shift (Granlund and Montgomery, "Division by
// invariant integers using multiplication", PLDI 1994, Thm. 4.2): with
// l = ceil(log2 d) and m = floor(2^(31+l) / d) + 1, m*d - 2^(31+l) <= d <= 2^l,
// hence floor(n / d) = floor(n * m / 2^(31+l)) for every such n, and m < 2^32.
struct FastDiv {
  uint32_t m;
  int sh;
};
inline FastDiv make_fastdiv(uint32_t d) {
  int l = 0;
  while ((1ull << l) < d) ++l;
  return FastDiv{(uint32_t)((1ull << (31 + l)) / d + 1), 31 + l};
}
#ifdef __CUDACC__
__device__ __forceinline__ int fdiv(int n, FastDiv f) {
  return (int)(((uint64_t)(uint32_t)n * f.m) >> f.sh);
}
#endif

// ---------------------------------------------------------------------------
// Parameters of the shift-GEMM kernels (FC and conv implicit GEMM).
// The GEMM view: rows = FC rows m or conv output pixels (n, oh, ow);
// columns = output features / channels; reduction = K or (c, r, s).
// ---------------------------------------------------------------------------
struct GemmParams {
  const int32_t* x;
  const uint8_t* blob;
  const int32_t* xcodes;    // nullable: expanded layout [ceil(cols/32)][kred][64]
  const int32_t* bias;      // nullable
  const int32_t* residual;  // nullable (conv, DS_RESIDUAL)
  int32_t* y;
  const uint32_t* amax_in;  // nullable: then the 64-bit path is taken
  uint32_t* amax_out;       // nullable
  int64_t rows;             // FC: M; conv: N*OH*OW
  int64_t kred;             // FC: K; conv: C*R*S
  int64_t cols;             // FC: N; conv: K
  int64_t n_chunks;
  int64_t off_nib, off_bits, off_cola, off_nnz;
  // conv geometry (unused by FC)
  int C, H, W, R, S, sh, sw, ph, pw, OH, OW;
  // implicit GEMM output placement (0: dense): output pixel (oh, ow) is stored
  // at (ys_h * oh + yph, ys_w * ow + ypw) of a yH x yW plane (one phase of a
  // strided layer's input gradient)
  int ys_h, ys_w, yph, ypw, yH, yW;
  uint32_t flags;
  // split reduction (conv, chained forward only): int64 partial sums of every
  // output; its first kSmallScratchBytes are zero on entry and on exit
  int64_t* split_acc;       // nullable
  size_t split_capacity;    // bytes available at split_acc
};

// Defined in shift_gemm.cu: up to kMaxGemmPhases implicit GEMMs (conv, no split) per launch.
constexpr int kMaxGemmPhases = 4;
cudaError_t launch_conv2d_shift_phases(const GemmParams* ps, int n, cudaStream_t st);
// Defined in conv_narrow.cu: stride-1 ConvShift with at most 8 output columns and at most 4 taps per row.
bool conv_narrow_supported(const GemmParams& p);
cudaError_t launch_conv_narrow(const GemmParams& p, cudaStream_t st);
// Launchers (defined in shift_gemm.cu).
cudaError_t launch_linear_shift(const GemmParams& p, cudaStream_t st);
// Defined in linear_cluster.cu (small batches: the reduction split over a thread-block cluster).
bool linear_cluster_preferred(const GemmParams& p);
cudaError_t launch_linear_cluster(const GemmParams& p, cudaStream_t st);
cudaError_t launch_conv2d_shift(const GemmParams& p, cudaStream_t st);
// Defined in conv_direct.cu.
bool conv_direct_supported(const GemmParams& p);
size_t conv_direct_split_bytes(const GemmParams& p);  // int64 scratch a split reduction would use (0: no split)
cudaError_t launch_conv2d_direct(const GemmParams& p, cudaStream_t st);
// Epilogue of a split reduction: y = ReLU?(sat32(sat32(split_acc + bias) + residual)), max|y|;
// re-zeroes the first kSmallScratchBytes of the scratch.
cudaError_t launch_split_finalize(const GemmParams& p, cudaStream_t st);
// Before a split launch: zeroes a scratch region larger than kSmallScratchBytes (smaller ones are zero).
constexpr size_t kSmallScratchBytes = 2u << 20;
cudaError_t prepare_split_scratch(const GemmParams& p, cudaStream_t st);
// Defined in conv_pointwise.cu (1x1 convolutions as a GEMM over pixels).
bool conv_pointwise_supported(const GemmParams& p);
size_t conv_pointwise_split_bytes(const GemmParams& p);
cudaError_t launch_conv2d_pointwise(const GemmParams& p, cudaStream_t st);
// Defined in api.cu: the split scratch of the kernel conv_launch would choose.
size_t conv_split_bytes(const GemmParams& p);
// Defined in linear_bf16.cu.
int64_t bf16_kpad(int64_t k_red);
cudaError_t launch_expand_bf16(const uint8_t* blob, int64_t n_out, int64_t k_red, uint16_t* out, cudaStream_t st);
cudaError_t launch_linear_bf16(const uint16_t* x, const uint16_t* w16, const float* bias, float* y, int64_t M,
                               int64_t K, int64_t N, uint32_t flags, cudaStream_t st);
int read_bf16_fault_flag();
void set_bf16_wait_cycles(long long cycles);
// Defined in chain_ops.cu.
cudaError_t launch_maxpool(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW, int R,
                           int S, int stride, int pad, cudaStream_t st);
cudaError_t launch_avgpool_floor(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW,
                                 int R, int S, int stride, cudaStream_t st);
// Defined in api.cu: launches after validation, with explicit amax slots.
ds_status check_weights(const ds_weights* w, int64_t n_out, int64_t k_red);
ds_status window_output(int H, int W, int R, int S, int stride_h, int stride_w, int pad_h, int pad_w, int* OH,
                        int* OW);
ds_status check_image(int C, int H, int W, int OH, int OW);
ds_status conv_launch(const int32_t* x, const ds_weights* w, const int32_t* bias, const int32_t* residual,
                      int32_t* y, int N, int C, int H, int W, int K, int R, int S, int stride, int pad,
                      uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out, cudaStream_t st,
                      int64_t* split_acc = nullptr, size_t split_capacity = 0);
GemmParams conv_params(const ds_weights* w, int N, int C, int H, int W, int K, int R, int S, int stride, int pad);
ds_status fc_launch(const int32_t* x, const ds_weights* w, const int32_t* bias, int32_t* y, int64_t M,
                    int64_t K, int64_t N, uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out,
                    cudaStream_t st);
// Defined in quantize.cu (DeepShift-Q codes from float weights, Q16.16 from float activations).
cudaError_t launch_quantize_weights(const float* w, int64_t n, int p_min, int8_t* s, int8_t* p, cudaStream_t st);
cudaError_t launch_quantize_q16(const float* x, int64_t n, int32_t* q, cudaStream_t st);
// Defined in specialize.cu (weight-specialised ConvShift compiled at run time).
ds_status specialize_conv(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride, int pad,
                          ds_specialized** out);
void specialized_dims(const ds_specialized* h, int* K, int* C, int* R, int* S, int* stride, int* pad);
cudaError_t launch_specialized(const ds_specialized* h, const int32_t* x, const int32_t* bias,
                               const int32_t* residual, int32_t* y, int N, int H, int W, int OH, int OW,
                               uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out, cudaStream_t st);
void destroy_specialized(ds_specialized* h);
// Defined in misc_kernels.cu.
// Streaming multiprocessors of the device this process uses, read once per
// process (one device per process); 0 when no device can be queried, in which
// case the grid heuristics plan no split reduction and no launch succeeds.
int sm_count();
cudaError_t launch_absmax(const int32_t* x, int64_t n, uint32_t* out, cudaStream_t st);
// bwd != nullptr: pack one phase of the input-gradient codes of forward codes
// [K][C][R][S]: bwd = {K, C, R, S, sh, sw, a, b, Th, Tw}; column c, index
// (k, t, u) reads code (k, c, a + sh (Th-1-t), b + sw (Tw-1-u)).
cudaError_t launch_pack(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red,
                        uint8_t* blob, cudaStream_t st, const int* bwd = nullptr);
cudaError_t launch_expand(const uint8_t* blob, int64_t n_out, int64_t k_red, int32_t* out, cudaStream_t st);

__host__ __device__ inline int64_t expanded_words(int64_t n_out, int64_t k_red) {
  return ((n_out + 31) / 32) * k_red * 64;
}

#ifdef __CUDACC__
// Asynchronous global -> shared copies of 4, 8 or 16 bytes; valid = false
// zero-fills the destination (source size 0).  4 and 8 bytes go through L1,
// 16 bytes bypass it.
__device__ __forceinline__ void cp_async4(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(gsrc), "r"(valid ? 4 : 0));
}
__device__ __forceinline__ void cp_async8(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;\n" ::"r"(d), "l"(gsrc), "r"(valid ? 8 : 0));
}
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(gsrc), "r"(valid ? 16 : 0));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
// Wait until at most N of this thread's committed copy groups are in flight.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}
__device__ __forceinline__ void cp_async_wait_all() { cp_async_wait<0>(); }
// Saturating int32 addition (the residual join) and |v| as an unsigned value.
__device__ __forceinline__ int32_t add_sat(int32_t a, int32_t b) {
  int32_t r;
  asm("add.sat.s32 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t uabs(int32_t v) { return v < 0 ? (uint32_t)0 - (uint32_t)v : (uint32_t)v; }

// Staging of the expanded codes of 64 columns (two 32-column blocks) and 16
// reduction indices per stage, by 128 threads: the stage is 512 16-byte
// pieces, and thread t copies the pieces at index kl = t / 16 and kl + 8 of
// both blocks, bytes 16 (t % 16) of the 64-word row, into
// cs[kl][block][64].  The pieces are the same at every stage, so the source
// address is computed once and advances by 16 indices per stage.
struct ExpandedCodeStager {
  const int32_t* src;  // (block 0, kl) at stage 0
  int64_t kp;          // kl's reduction index at stage 0
  int64_t kred_words;  // words between the two blocks' rows of one index: kred * 64
  bool b1;             // block 1 exists
  __device__ __forceinline__ ExpandedCodeStager(const int32_t* xcodes, int64_t cols, int64_t kred, int64_t col0,
                                                int64_t kbeg) {
    const int t = threadIdx.x;
    const int64_t cb = col0 / 32;
    b1 = cb + 1 < (cols + 31) / 32;
    kp = kbeg + (t >> 4);
    kred_words = kred * 64;
    src = xcodes != nullptr ? xcodes + (cb * kred + kp) * 64 + (t & 15) * 4 : xcodes;
  }
  // stage st with both blocks present and all 16 indices inside the reduction: no checks
  __device__ __forceinline__ void stage_full(int32_t* cs, int st) const {
    const int t = threadIdx.x;
    const int32_t* s = src + (int64_t)st * 16 * 64;
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(cs + (t >> 4) * 128 + (t & 15) * 4);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int kl8 = (u & 1) * 8, b = u >> 1;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d + (uint32_t)(kl8 * 128 + b * 64) * 4),
                   "l"(s + kl8 * 64 + b * kred_words));
    }
  }
  // stage st (indices kbeg + 16 st ..) into cs; zero fill past kred and for an absent block
  __device__ __forceinline__ void stage(const int32_t* xcodes, int64_t kred, int32_t* cs, int st) const {
    const int t = threadIdx.x;
    const int64_t k = kp + (int64_t)st * 16;
    const int32_t* s = src + (int64_t)st * 16 * 64;
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(cs + (t >> 4) * 128 + (t & 15) * 4);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int kl8 = (u & 1) * 8, b = u >> 1;
      const bool ok = k + kl8 < kred && (b == 0 || b1);
      const int32_t* g = ok ? s + kl8 * 64 + b * kred * 64 : xcodes;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d + (uint32_t)(kl8 * 128 + b * 64) * 4),
                   "l"(g), "r"(ok ? 16 : 0));
    }
  }
};
#endif

}  // namespace ds
