// Shared definitions of the DeepShift CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "deepshift.h"

namespace ds {

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
// Defined in chain_ops.cu.
cudaError_t launch_maxpool(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW, int R,
                           int S, int stride, int pad, cudaStream_t st);
cudaError_t launch_avgpool_floor(const int32_t* x, int32_t* y, int64_t planes, int H, int W, int OH, int OW,
                                 int R, int S, int stride, cudaStream_t st);
// Defined in api.cu: launches after validation, with explicit amax slots.
ds_status check_weights(const ds_weights* w, int64_t n_out, int64_t k_red);
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
// Defined in misc_kernels.cu.
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

}  // namespace ds
