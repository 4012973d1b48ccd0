// C ABI entry points of the shift operators (Eq. 3), the code conversion
// (Eq. 4-6) and the input gradient (Eq. 7): argument validation, then
// stream-ordered launches.
// Nothing is launched and no output is written when validation fails.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <initializer_list>

#include "ds_common.cuh"

namespace ds {

// The last error of the calling thread, in a fixed buffer: recording an error
// never allocates, so no entry point can fail (or throw) while reporting one.
static thread_local char g_last_error[512];

void set_error(const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  memcpy(g_last_error, buf, sizeof(buf));
}

void clear_error() { g_last_error[0] = '\0'; }

ds_status fail(ds_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  memcpy(g_last_error, buf, sizeof(buf));
  return st;
}

ds_status cuda_check(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return DS_OK;
  return fail(DS_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// Byte size of an int32 tensor with the given positive extents, or -1 when it
// exceeds 2^62 bytes: no buffer is that large, and the bound keeps every
// element offset the kernels form inside int64.
static int64_t int32_tensor_bytes(std::initializer_list<int64_t> dims) {
  int64_t n = sizeof(int32_t);
  for (int64_t d : dims)
    if (d <= 0 || __builtin_mul_overflow(n, d, &n) || n > (int64_t(1) << 62)) return -1;
  return n;
}

// A code matrix is accepted when n_out <= 2^31, k_red <= k_max and it holds
// at most 2^48 codes, which keeps every size derived from it (packed,
// expanded, bf16) far inside 64 bits.
static bool code_matrix_in_range(int64_t n_out, int64_t k_red, int64_t k_max) {
  return n_out > 0 && k_red > 0 && n_out <= (int64_t(1) << 31) && k_red <= k_max &&
         k_red <= (int64_t(1) << 48) / n_out;
}

// True when the byte ranges [a, a + na) and [b, b + nb) intersect.  The ends
// are formed as integers, so no pointer is moved past its buffer.
static bool ranges_overlap(const void* a, int64_t na, const void* b, int64_t nb) {
  const uintptr_t ua = reinterpret_cast<uintptr_t>(a), ub = reinterpret_cast<uintptr_t>(b);
  return ua < ub + static_cast<uintptr_t>(nb) && ub < ua + static_cast<uintptr_t>(na);
}

// Output size of a window (convolution or pooling) over a zero-padded image,
// formed in 64 bits: positive extents and strides, non-negative pads, a
// window no larger than the padded image, and a padded extent within int32.
ds_status window_output(int H, int W, int R, int S, int stride_h, int stride_w, int pad_h, int pad_w, int* OH,
                        int* OW) {
  if (H <= 0 || W <= 0 || R <= 0 || S <= 0) return fail(DS_ERR_SHAPE, "H, W, R and S must be positive");
  if (stride_h <= 0 || stride_w <= 0 || pad_h < 0 || pad_w < 0)
    return fail(DS_ERR_SHAPE, "strides must be positive and pads non-negative");
  const int64_t hp = (int64_t)H + 2 * (int64_t)pad_h, wp = (int64_t)W + 2 * (int64_t)pad_w;
  if (hp < R || wp < S) return fail(DS_ERR_SHAPE, "kernel larger than padded input");
  if (hp > INT32_MAX || wp > INT32_MAX) return fail(DS_ERR_UNSUPPORTED, "padded input larger than 2^31 - 1");
  *OH = (int)((hp - R) / stride_h + 1);
  *OW = (int)((wp - S) / stride_w + 1);
  return DS_OK;
}

// Per-image limits of the convolution and pooling kernels, which index
// within one image in 32 bits: C x H x W <= 2^31 inputs, OH x OW <= 2^30
// outputs per plane.
ds_status check_image(int C, int H, int W, int OH, int OW) {
  const int64_t xb = int32_tensor_bytes({C, H, W});
  if (xb < 0 || xb > (int64_t(4) << 31) || (int64_t)OH * OW > (int64_t)1 << 30)
    return fail(DS_ERR_UNSUPPORTED, "image too large");
  return DS_OK;
}

// Checks a descriptor filled by ds_pack_shift_weights against the call's dims.
ds_status check_weights(const ds_weights* w, int64_t n_out, int64_t k_red) {
  if (w == nullptr) return fail(DS_ERR_INVALID_ARG, "weights descriptor is NULL");
  if (w->magic != DS_WEIGHTS_MAGIC || w->format != DS_FORMAT_PLANES6)
    return fail(DS_ERR_INVALID_ARG, "weights descriptor was not filled by ds_pack_shift_weights");
  if (w->packed == nullptr) return fail(DS_ERR_INVALID_ARG, "weights descriptor has no blob");
  if (w->n_out != n_out || w->k_red != k_red)
    return fail(DS_ERR_SHAPE, "weights are %lld x %lld, call needs %lld x %lld", (long long)w->n_out,
                (long long)w->k_red, (long long)n_out, (long long)k_red);
  if (ds_packed_weight_bytes(n_out, k_red) == 0)
    return fail(DS_ERR_UNSUPPORTED, "a %lld x %lld code matrix is outside the supported range", (long long)n_out,
                (long long)k_red);
  const BlobLayout L = blob_layout(n_out, k_red);
  if (w->n_chunks != L.n_chunks || w->packed_bytes < (size_t)L.total)
    return fail(DS_ERR_INVALID_ARG, "weights descriptor is inconsistent with its dims");
  if ((reinterpret_cast<uintptr_t>(w->packed) & 255) != 0)
    return fail(DS_ERR_ALIGNMENT, "packed blob must be 256-byte aligned");
  return DS_OK;
}

static void fill_blob_offsets(GemmParams& p, const ds_weights* w) {
  const BlobLayout L = blob_layout(w->n_out, w->k_red);
  p.blob = static_cast<const uint8_t*>(w->packed);
  p.xcodes = (w->expanded != nullptr &&
              w->expanded_bytes >= (size_t)expanded_words(w->n_out, w->k_red) * sizeof(int32_t))
                 ? static_cast<const int32_t*>(w->expanded)
                 : nullptr;
  p.n_chunks = L.n_chunks;
  p.off_nib = L.nib;
  p.off_bits = L.bits;
  p.off_cola = L.col_a;
  p.off_nnz = L.nnz;
}

// Resolves the amax slots: computes max|x| into amax_io[0] unless the caller
// provided it, and zeroes amax_io[1] when the call reports the output amax.
static ds_status prepare_amax(const int32_t* x, int64_t nx, uint32_t flags, uint32_t* amax_io,
                              cudaStream_t st, GemmParams& p) {
  p.amax_in = nullptr;
  p.amax_out = nullptr;
  if (amax_io == nullptr) return DS_OK;
  if (!(flags & DS_AMAX_IN)) {
    ds_status s = cuda_check(launch_absmax(x, nx, amax_io, st), "absmax pre-pass");
    if (s != DS_OK) return s;
  }
  p.amax_in = amax_io;
  if (flags & DS_AMAX_OUT) {
    ds_status s = cuda_check(cudaMemsetAsync(amax_io + 1, 0, sizeof(uint32_t), st), "amax_out reset");
    if (s != DS_OK) return s;
    p.amax_out = amax_io + 1;
  }
  return DS_OK;
}

GemmParams conv_params(const ds_weights* w, int N, int C, int H, int W, int K, int R, int S, int stride,
                       int pad) {
  GemmParams p{};
  p.OH = (H + 2 * pad - R) / stride + 1;
  p.OW = (W + 2 * pad - S) / stride + 1;
  p.rows = (int64_t)N * p.OH * p.OW;
  p.kred = (int64_t)C * R * S;
  p.cols = K;
  p.C = C;
  p.H = H;
  p.W = W;
  p.R = R;
  p.S = S;
  p.sh = stride;
  p.sw = stride;
  p.ph = pad;
  p.pw = pad;
  fill_blob_offsets(p, w);
  return p;
}

ds_status conv_launch(const int32_t* x, const ds_weights* w, const int32_t* bias, const int32_t* residual,
                      int32_t* y, int N, int C, int H, int W, int K, int R, int S, int stride, int pad,
                      uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out, cudaStream_t st,
                      int64_t* split_acc, size_t split_capacity) {
  GemmParams p = conv_params(w, N, C, H, W, K, R, S, stride, pad);
  p.x = x;
  p.bias = bias;
  p.residual = (flags & DS_RESIDUAL) ? residual : nullptr;
  p.y = y;
  p.flags = flags;
  p.amax_in = amax_in;
  p.amax_out = amax_out;
  p.split_acc = split_acc;
  p.split_capacity = split_capacity;
  if (!(flags & DS_CONV_IM2COL)) {
    if (conv_pointwise_supported(p)) return cuda_check(launch_conv2d_pointwise(p, st), "conv2d_shift (pointwise) launch");
    if (conv_direct_supported(p)) return cuda_check(launch_conv2d_direct(p, st), "conv2d_shift (direct) launch");
  }
  p.split_acc = nullptr;
  return cuda_check(launch_conv2d_shift(p, st), "conv2d_shift (implicit GEMM) launch");
}

size_t conv_split_bytes(const GemmParams& p) {
  if (conv_pointwise_supported(p)) return conv_pointwise_split_bytes(p);
  return conv_direct_split_bytes(p);
}

// LinearShift kernel choice: small batches split the reduction over a
// thread-block cluster, large ones run the 128 x 64-tile shift GEMM.
static ds_status launch_fc(const GemmParams& p, cudaStream_t st) {
  if (linear_cluster_preferred(p)) return cuda_check(launch_linear_cluster(p, st), "linear_shift (cluster) launch");
  return cuda_check(launch_linear_shift(p, st), "linear_shift launch");
}

ds_status fc_launch(const int32_t* x, const ds_weights* w, const int32_t* bias, int32_t* y, int64_t M,
                    int64_t K, int64_t N, uint32_t flags, const uint32_t* amax_in, uint32_t* amax_out,
                    cudaStream_t st) {
  GemmParams p{};
  p.x = x;
  p.bias = bias;
  p.residual = nullptr;
  p.y = y;
  p.rows = M;
  p.kred = K;
  p.cols = N;
  p.flags = flags;
  fill_blob_offsets(p, w);
  p.amax_in = amax_in;
  p.amax_out = amax_out;
  return launch_fc(p, st);
}

ds_status pack_finish(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red, void* packed, size_t need,
                      ds_weights* desc, cudaStream_t st, const int* bwd);

// Taps r = a, a + stride, ... < R of tap phase a (the input-gradient decomposition of a strided layer).
static int phase_taps(int R, int stride, int a) { return a < R ? (R - 1 - a) / stride + 1 : 0; }

constexpr uint32_t kKnownFlags =
    DS_RELU | DS_AMAX_IN | DS_AMAX_OUT | DS_RESIDUAL | DS_FORCE_INT64 | DS_CONV_IM2COL;

}  // namespace ds

using namespace ds;

extern "C" {

const char* ds_last_error(void) { return g_last_error; }

int ds_version(void) { return 100; }

size_t ds_abi_struct_size(int which) {
  return which == 0 ? sizeof(ds_weights) : (which == 1 ? sizeof(ds_layer) : 0);
}

size_t ds_packed_weight_bytes(int64_t n_out, int64_t k_red) {
  if (!code_matrix_in_range(n_out, k_red, int64_t(1) << 40)) return 0;
  return (size_t)blob_layout(n_out, k_red).total;
}

ds_status ds_pack_shift_weights(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red,
                                void* packed, size_t packed_bytes, ds_weights* desc, void* stream) {
  NvtxRange nvtx_range("ds_pack_shift_weights");
  clear_error();
  if (!s || !p || !packed || !desc) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n_out <= 0 || k_red <= 0) return fail(DS_ERR_SHAPE, "n_out and k_red must be positive");
  const size_t need = ds_packed_weight_bytes(n_out, k_red);
  if (need == 0) return fail(DS_ERR_UNSUPPORTED, "code matrix too large");
  if (packed_bytes < need)
    return fail(DS_ERR_BUFFER_TOO_SMALL, "packed buffer has %zu bytes, needs %zu", packed_bytes, need);
  if ((reinterpret_cast<uintptr_t>(packed) & 255) != 0)
    return fail(DS_ERR_ALIGNMENT, "packed buffer must be 256-byte aligned");
  return pack_finish(s, p, n_out, k_red, packed, need, desc, static_cast<cudaStream_t>(stream), nullptr);
}

}  // extern "C"

namespace ds {
// Launches the pack, waits for it and fills the descriptor (shared by the
// forward and the input-gradient packing).
ds_status pack_finish(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red, void* packed, size_t need,
                      ds_weights* desc, cudaStream_t st, const int* bwd) {
  uint8_t* blob = static_cast<uint8_t*>(packed);
  ds_status r = cuda_check(launch_pack(s, p, n_out, k_red, blob, st, bwd), "pack launch");
  if (r != DS_OK) return r;
  BlobHeader h;
  r = cuda_check(cudaMemcpyAsync(&h, blob, sizeof(h), cudaMemcpyDeviceToHost, st), "header read");
  if (r != DS_OK) return r;
  r = cuda_check(cudaStreamSynchronize(st), "pack synchronise");
  if (r != DS_OK) return r;
  if (h.invalid_count != 0)
    return fail(DS_ERR_CODE_RANGE, "%u codes outside s in {-1,0,1} or p in [-15,0]", h.invalid_count);
  desc->magic = DS_WEIGHTS_MAGIC;
  desc->format = DS_FORMAT_PLANES6;
  desc->n_out = n_out;
  desc->k_red = k_red;
  desc->n_chunks = h.n_chunks;
  desc->packed = packed;
  desc->packed_bytes = need;
  desc->a_max = h.a_max;
  desc->nnz_max = h.nnz_max;
  desc->reserved = 0;
  desc->expanded = nullptr;
  desc->expanded_bytes = 0;
  desc->weights_bf16 = nullptr;
  desc->weights_bf16_bytes = 0;
  return DS_OK;
}
}  // namespace ds

extern "C" {

size_t ds_packed_weight_bytes_backward(int K, int C, int R, int S, int stride_h, int stride_w) {
  if (K <= 0 || C <= 0 || R <= 0 || S <= 0 || stride_h <= 0 || stride_w <= 0) return 0;
  size_t total = 0;
  for (int a = 0; a < stride_h; ++a)
    for (int b = 0; b < stride_w; ++b) {
      const int th = phase_taps(R, stride_h, a), tw = phase_taps(S, stride_w, b);
      if (th == 0 || tw == 0) continue;
      const size_t one = ds_packed_weight_bytes(C, (int64_t)K * th * tw);
      if (one == 0) return 0;
      total += (one + 255) / 256 * 256;
    }
  return total;
}

ds_status ds_pack_shift_weights_backward(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride_h,
                                         int stride_w, void* packed, size_t packed_bytes, ds_weights* desc,
                                         void* stream) {
  NvtxRange nvtx_range("ds_pack_shift_weights_backward");
  clear_error();
  if (!s || !p || !packed || !desc) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (K <= 0 || C <= 0 || R <= 0 || S <= 0) return fail(DS_ERR_SHAPE, "K, C, R and S must be positive");
  if (stride_h <= 0 || stride_w <= 0 || stride_h > 16 || stride_w > 16)
    return fail(DS_ERR_SHAPE, "strides must be in [1, 16]");
  const size_t need = ds_packed_weight_bytes_backward(K, C, R, S, stride_h, stride_w);
  if (need == 0) return fail(DS_ERR_UNSUPPORTED, "code matrix too large");
  if (packed_bytes < need)
    return fail(DS_ERR_BUFFER_TOO_SMALL, "packed buffer has %zu bytes, needs %zu", packed_bytes, need);
  if ((reinterpret_cast<uintptr_t>(packed) & 255) != 0)
    return fail(DS_ERR_ALIGNMENT, "packed buffer must be 256-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  size_t off = 0;
  for (int a = 0; a < stride_h; ++a)
    for (int b = 0; b < stride_w; ++b) {
      ds_weights& d = desc[a * stride_w + b];
      const int th = phase_taps(R, stride_h, a), tw = phase_taps(S, stride_w, b);
      if (th == 0 || tw == 0) {  // a phase no tap reaches: its input-gradient positions are zero
        d = ds_weights{};
        d.magic = DS_WEIGHTS_MAGIC;
        d.format = DS_FORMAT_PLANES6;
        d.n_out = C;
        d.k_red = 0;
        continue;
      }
      const int64_t k_red = (int64_t)K * th * tw;
      const size_t one = ds_packed_weight_bytes(C, k_red);
      const int map[10] = {K, C, R, S, stride_h, stride_w, a, b, th, tw};
      ds_status r = pack_finish(s, p, C, k_red, static_cast<unsigned char*>(packed) + off, one, &d, st, map);
      if (r != DS_OK) return r;
      off += (one + 255) / 256 * 256;
    }
  return DS_OK;
}

size_t ds_expanded_weight_bytes(int64_t n_out, int64_t k_red) {
  if (!code_matrix_in_range(n_out, k_red, int64_t(1) << 36)) return 0;
  return (size_t)expanded_words(n_out, k_red) * sizeof(int32_t);
}

ds_status ds_expand_shift_weights(ds_weights* w, void* expanded, size_t expanded_bytes, void* stream) {
  NvtxRange nvtx_range("ds_expand_shift_weights");
  clear_error();
  if (w == nullptr || expanded == nullptr) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  ds_status r = check_weights(w, w->n_out, w->k_red);
  if (r != DS_OK) return r;
  const size_t need = ds_expanded_weight_bytes(w->n_out, w->k_red);
  if (need == 0) return fail(DS_ERR_UNSUPPORTED, "code matrix too large to expand");
  if (expanded_bytes < need)
    return fail(DS_ERR_BUFFER_TOO_SMALL, "expanded buffer has %zu bytes, needs %zu", expanded_bytes, need);
  if (!aligned16(expanded)) return fail(DS_ERR_ALIGNMENT, "expanded buffer must be 16-byte aligned");
  r = cuda_check(launch_expand(static_cast<const uint8_t*>(w->packed), w->n_out, w->k_red,
                               static_cast<int32_t*>(expanded), static_cast<cudaStream_t>(stream)),
                 "expand launch");
  if (r != DS_OK) return r;
  w->expanded = expanded;
  w->expanded_bytes = need;
  return DS_OK;
}

size_t ds_bf16_weight_bytes(int64_t n_out, int64_t k_red) {
  if (!code_matrix_in_range(n_out, k_red, int64_t(1) << 36)) return 0;
  return (size_t)(n_out * bf16_kpad(k_red) * 2 + 255) / 256 * 256;
}

ds_status ds_expand_shift_weights_bf16(ds_weights* w, void* buf, size_t bytes, void* stream) {
  NvtxRange nvtx_range("ds_expand_shift_weights_bf16");
  clear_error();
  if (w == nullptr || buf == nullptr) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  ds_status r = check_weights(w, w->n_out, w->k_red);
  if (r != DS_OK) return r;
  const size_t need = ds_bf16_weight_bytes(w->n_out, w->k_red);
  if (need == 0) return fail(DS_ERR_UNSUPPORTED, "code matrix too large");
  if (bytes < need) return fail(DS_ERR_BUFFER_TOO_SMALL, "bf16 buffer has %zu bytes, needs %zu", bytes, need);
  if (!aligned16(buf)) return fail(DS_ERR_ALIGNMENT, "bf16 buffer must be 16-byte aligned");
  r = cuda_check(launch_expand_bf16(static_cast<const uint8_t*>(w->packed), w->n_out, w->k_red,
                                    static_cast<uint16_t*>(buf), static_cast<cudaStream_t>(stream)),
                 "bf16 expand launch");
  if (r != DS_OK) return r;
  w->weights_bf16 = buf;
  w->weights_bf16_bytes = need;
  return DS_OK;
}

ds_status ds_linear_shift_bf16(const uint16_t* x, const ds_weights* w, const float* bias, float* y, int64_t M,
                               int64_t K, int64_t N, uint32_t flags, void* stream) {
  NvtxRange nvtx_range("ds_linear_shift_bf16");
  clear_error();
  if (!x || !y) return fail(DS_ERR_INVALID_ARG, "NULL x or y");
  if (M <= 0 || K <= 0 || N <= 0) return fail(DS_ERR_SHAPE, "M, K and N must be positive");
  if (M > ((int64_t)1 << 31) - 256 || N > ((int64_t)1 << 31) - 256) return fail(DS_ERR_UNSUPPORTED, "M or N too large");
  if (flags & ~DS_RELU) return fail(DS_ERR_INVALID_ARG, "only DS_RELU applies to the float variant");
  if (!aligned16(x) || !aligned16(y)) return fail(DS_ERR_ALIGNMENT, "x and y must be 16-byte aligned");
  if (K % 8 != 0) return fail(DS_ERR_UNSUPPORTED, "K must be a multiple of 8 (16-byte bf16 rows)");
  ds_status r = check_weights(w, N, K);
  if (r != DS_OK) return r;
  if (w->weights_bf16 == nullptr || w->weights_bf16_bytes < ds_bf16_weight_bytes(N, K))
    return fail(DS_ERR_UNSUPPORTED, "bf16 weights missing: call ds_expand_shift_weights_bf16 first");
  return cuda_check(launch_linear_bf16(x, static_cast<const uint16_t*>(w->weights_bf16), bias, y, M, K, N, flags,
                                       static_cast<cudaStream_t>(stream)),
                    "linear_shift_bf16 launch");
}

int ds_bf16_fault_flag(void) { return read_bf16_fault_flag(); }

void ds_bf16_set_wait_limit(long long cycles) { set_bf16_wait_cycles(cycles); }

ds_status ds_linear_shift_backward_x(const int32_t* dy, const ds_weights* w_bwd, int32_t* dx, int64_t M, int64_t K,
                                     int64_t N, uint32_t flags, uint32_t* amax_io, void* stream) {
  NvtxRange nvtx_range("ds_linear_shift_backward_x");
  clear_error();
  if (flags & ~(DS_AMAX_IN | DS_AMAX_OUT | DS_FORCE_INT64))
    return fail(DS_ERR_INVALID_ARG, "only DS_AMAX_IN, DS_AMAX_OUT and DS_FORCE_INT64 apply to a gradient");
  // dX [M][K] = dY [M][N] times the input-gradient codes (K columns, reduction N)
  return ds_linear_shift(dy, w_bwd, nullptr, dx, M, N, K, flags, amax_io, stream);
}

ds_status ds_conv2d_shift_backward_x(const int32_t* dy, const ds_weights* w_bwd, int32_t* dx, int N, int C, int H,
                                     int W, int K, int R, int S, int stride_h, int stride_w, int pad_h, int pad_w,
                                     uint32_t flags, uint32_t* amax_io, void* stream) {
  NvtxRange nvtx_range("ds_conv2d_shift_backward_x");
  clear_error();
  if (!dy || !dx || !w_bwd) return fail(DS_ERR_INVALID_ARG, "NULL dy, dx or weights");
  if (N <= 0 || C <= 0 || H <= 0 || W <= 0 || K <= 0 || R <= 0 || S <= 0)
    return fail(DS_ERR_SHAPE, "N, C, H, W, K, R, S must be positive");
  if (stride_h <= 0 || stride_w <= 0 || stride_h > 16 || stride_w > 16 || pad_h < 0 || pad_w < 0)
    return fail(DS_ERR_SHAPE, "strides must be in [1, 16] and pads non-negative");
  int OH = 0, OW = 0;
  ds_status rg = window_output(H, W, R, S, stride_h, stride_w, pad_h, pad_w, &OH, &OW);
  if (rg != DS_OK) return rg;
  if (flags & ~(DS_AMAX_IN | DS_AMAX_OUT | DS_FORCE_INT64 | DS_CONV_IM2COL))
    return fail(DS_ERR_INVALID_ARG, "only DS_AMAX_IN, DS_AMAX_OUT, DS_FORCE_INT64, DS_CONV_IM2COL apply here");
  if ((flags & (DS_AMAX_IN | DS_AMAX_OUT)) && amax_io == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_AMAX_IN / DS_AMAX_OUT need amax_io");
  // one descriptor per tap phase (a, b), as ds_pack_shift_weights_backward fills them
  bool empty_phase = false;
  for (int a = 0; a < stride_h; ++a)
    for (int b = 0; b < stride_w; ++b) {
      const ds_weights& d = w_bwd[a * stride_w + b];
      const int th = phase_taps(R, stride_h, a), tw = phase_taps(S, stride_w, b);
      if (th == 0 || tw == 0) {
        if (d.magic != DS_WEIGHTS_MAGIC || d.n_out != C || d.k_red != 0)
          return fail(DS_ERR_INVALID_ARG, "phase (%d, %d): descriptor does not match the layer", a, b);
        empty_phase = true;
        continue;
      }
      ds_status r = check_weights(&d, C, (int64_t)K * th * tw);
      if (r != DS_OK) return r;
    }
  // stride 1: the forward ConvShift of dY with the rot180 / transposed codes and padding R-1-pad
  if (stride_h == 1 && stride_w == 1 && pad_h <= R - 1 && pad_w <= S - 1 && !(flags & DS_CONV_IM2COL))
    return ds_conv2d_shift(dy, w_bwd, nullptr, nullptr, dx, N, K, OH, OW, C, R, S, 1, 1, R - 1 - pad_h,
                           S - 1 - pad_w, flags, amax_io, stream);
  if (!aligned16(dy) || !aligned16(dx)) return fail(DS_ERR_ALIGNMENT, "dy and dx must be 16-byte aligned");
  // dY is this pass's input image (K x OH x OW) and dX its output plane (H x W)
  ds_status ri = check_image(K, OH, OW, H, W);
  if (ri != DS_OK) return ri;
  const int64_t yb = int32_tensor_bytes({N, K, OH, OW}), xb = int32_tensor_bytes({N, C, H, W});
  if (xb < 0 || yb < 0) return fail(DS_ERR_UNSUPPORTED, "dx or dy larger than 2^62 bytes");
  if (ranges_overlap(dx, xb, dy, yb)) return fail(DS_ERR_INVALID_ARG, "dx must not overlap dy");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  GemmParams base{};
  base.flags = flags & ~DS_CONV_IM2COL;
  ds_status r = prepare_amax(dy, yb / (int64_t)sizeof(int32_t), flags, amax_io, st, base);
  if (r != DS_OK) return r;
  if (empty_phase) {
    r = cuda_check(cudaMemsetAsync(dx, 0, (size_t)xb, st), "dx reset");
    if (r != DS_OK) return r;
  }
  // output phase (rh, rw): dX rows rh, rh + sh, ...; they receive the taps r = a + sh t with
  // a = (rh + pad_h) mod sh, reading gradient row i' + c_h - t (i = sh i' + rh, c_h = (rh + pad_h - a) / sh):
  // a stride-1 correlation of dY with the phase's Th x Tw sub-kernel and padding Th - 1 - c_h
  // the implicit-GEMM phases go out kMaxGemmPhases per launch (each alone fills few SMs)
  GemmParams gemm_phases[kMaxGemmPhases];
  int n_gemm = 0;
  for (int rh = 0; rh < stride_h && rh < H; ++rh)
    for (int rw = 0; rw < stride_w && rw < W; ++rw) {
      const int a = (rh + pad_h) % stride_h, b = (rw + pad_w) % stride_w;
      const int th = phase_taps(R, stride_h, a), tw = phase_taps(S, stride_w, b);
      if (th == 0 || tw == 0) continue;
      const int ch = (rh + pad_h - a) / stride_h, cw = (rw + pad_w - b) / stride_w;
      GemmParams p = base;
      p.x = dy;
      p.y = dx;
      p.C = K;
      p.H = OH;
      p.W = OW;
      p.R = th;
      p.S = tw;
      p.sh = 1;
      p.sw = 1;
      p.ph = th - 1 - ch;
      p.pw = tw - 1 - cw;
      p.OH = (H - rh + stride_h - 1) / stride_h;
      p.OW = (W - rw + stride_w - 1) / stride_w;
      p.rows = (int64_t)N * p.OH * p.OW;
      p.kred = (int64_t)K * th * tw;
      p.cols = C;
      p.ys_h = stride_h;
      p.ys_w = stride_w;
      p.yph = rh;
      p.ypw = rw;
      p.yH = H;
      p.yW = W;
      fill_blob_offsets(p, &w_bwd[a * stride_w + b]);
      // few columns (the gradient of a layer with few input channels): a thread per 4 pixels and all columns;
      // DS_CONV_IM2COL keeps the implicit GEMM (testing / comparison)
      if (conv_narrow_supported(p) && !(flags & DS_CONV_IM2COL)) {
        r = cuda_check(launch_conv_narrow(p, st), "conv2d_shift_backward_x (narrow) launch");
        if (r != DS_OK) return r;
      } else {
        gemm_phases[n_gemm++] = p;
        if (n_gemm == kMaxGemmPhases) {
          r = cuda_check(launch_conv2d_shift_phases(gemm_phases, n_gemm, st),
                         "conv2d_shift_backward_x (implicit GEMM) launch");
          if (r != DS_OK) return r;
          n_gemm = 0;
        }
      }
    }
  if (n_gemm > 0) {
    r = cuda_check(launch_conv2d_shift_phases(gemm_phases, n_gemm, st),
                   "conv2d_shift_backward_x (implicit GEMM) launch");
    if (r != DS_OK) return r;
  }
  return DS_OK;
}

ds_status ds_quantize_shift_weights(const float* w, int64_t n, int p_min, int8_t* s, int8_t* p, void* stream) {
  NvtxRange nvtx_range("ds_quantize_shift_weights");
  clear_error();
  if (!w || !s || !p) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n <= 0) return fail(DS_ERR_SHAPE, "n must be positive");
  if (p_min < -15 || p_min > 0) return fail(DS_ERR_INVALID_ARG, "p_min %d outside [-15, 0]", p_min);
  if ((reinterpret_cast<uintptr_t>(w) & 3) != 0) return fail(DS_ERR_ALIGNMENT, "w must be 4-byte aligned");
  return cuda_check(launch_quantize_weights(w, n, p_min, s, p, static_cast<cudaStream_t>(stream)),
                    "quantize_shift_weights launch");
}

ds_status ds_quantize_q16(const float* x, int64_t n, int32_t* q, void* stream) {
  NvtxRange nvtx_range("ds_quantize_q16");
  clear_error();
  if (!x || !q) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n <= 0) return fail(DS_ERR_SHAPE, "n must be positive");
  if ((reinterpret_cast<uintptr_t>(x) & 3) != 0 || (reinterpret_cast<uintptr_t>(q) & 3) != 0)
    return fail(DS_ERR_ALIGNMENT, "x and q must be 4-byte aligned");
  return cuda_check(launch_quantize_q16(x, n, q, static_cast<cudaStream_t>(stream)), "quantize_q16 launch");
}

ds_status ds_absmax(const int32_t* x, int64_t n, uint32_t* amax, void* stream) {
  NvtxRange nvtx_range("ds_absmax");
  clear_error();
  if (!x || !amax) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  if (n <= 0) return fail(DS_ERR_SHAPE, "n must be positive");
  return cuda_check(launch_absmax(x, n, amax, static_cast<cudaStream_t>(stream)), "absmax launch");
}

ds_status ds_linear_shift(const int32_t* x, const ds_weights* w, const int32_t* bias, int32_t* y,
                          int64_t M, int64_t K, int64_t N, uint32_t flags, uint32_t* amax_io,
                          void* stream) {
  NvtxRange nvtx_range("ds_linear_shift");
  clear_error();
  if (!x || !y) return fail(DS_ERR_INVALID_ARG, "NULL x or y");
  if (M <= 0 || K <= 0 || N <= 0) return fail(DS_ERR_SHAPE, "M, K and N must be positive");
  if (M > (int64_t(1) << 40) || N > 65535LL * 64) return fail(DS_ERR_UNSUPPORTED, "M or N too large");
  if (flags & ~kKnownFlags) return fail(DS_ERR_INVALID_ARG, "unknown flag bits 0x%x", flags & ~kKnownFlags);
  if (flags & (DS_RESIDUAL | DS_CONV_IM2COL))
    return fail(DS_ERR_INVALID_ARG, "DS_RESIDUAL / DS_CONV_IM2COL apply to ds_conv2d_shift only");
  if ((flags & (DS_AMAX_IN | DS_AMAX_OUT)) && amax_io == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_AMAX_IN / DS_AMAX_OUT need amax_io");
  if (!aligned16(x) || !aligned16(y)) return fail(DS_ERR_ALIGNMENT, "x and y must be 16-byte aligned");
  ds_status r = check_weights(w, N, K);
  if (r != DS_OK) return r;
  const int64_t xb = int32_tensor_bytes({M, K}), yb = int32_tensor_bytes({M, N});
  if (xb < 0 || yb < 0) return fail(DS_ERR_UNSUPPORTED, "x or y larger than 2^62 bytes");
  if (ranges_overlap(x, xb, y, yb)) return fail(DS_ERR_INVALID_ARG, "y must not overlap x");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  GemmParams p{};
  p.x = x;
  p.bias = bias;
  p.residual = nullptr;
  p.y = y;
  p.rows = M;
  p.kred = K;
  p.cols = N;
  p.flags = flags;
  fill_blob_offsets(p, w);
  r = prepare_amax(x, M * K, flags, amax_io, st, p);
  if (r != DS_OK) return r;
  return launch_fc(p, st);
}

ds_status ds_conv2d_shift(const int32_t* x, const ds_weights* w, const int32_t* bias,
                          const int32_t* residual, int32_t* y, int N, int C, int H, int W, int K,
                          int R, int S, int stride_h, int stride_w, int pad_h, int pad_w,
                          uint32_t flags, uint32_t* amax_io, void* stream) {
  NvtxRange nvtx_range("ds_conv2d_shift");
  clear_error();
  if (!x || !y) return fail(DS_ERR_INVALID_ARG, "NULL x or y");
  if (N <= 0 || C <= 0 || H <= 0 || W <= 0 || K <= 0 || R <= 0 || S <= 0)
    return fail(DS_ERR_SHAPE, "N, C, H, W, K, R, S must be positive");
  int OH = 0, OW = 0;
  ds_status r = window_output(H, W, R, S, stride_h, stride_w, pad_h, pad_w, &OH, &OW);
  if (r != DS_OK) return r;
  if (flags & ~kKnownFlags) return fail(DS_ERR_INVALID_ARG, "unknown flag bits 0x%x", flags & ~kKnownFlags);
  if ((flags & DS_RESIDUAL) && residual == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_RESIDUAL needs a residual tensor");
  if ((flags & (DS_AMAX_IN | DS_AMAX_OUT)) && amax_io == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_AMAX_IN / DS_AMAX_OUT need amax_io");
  if (!aligned16(x) || !aligned16(y)) return fail(DS_ERR_ALIGNMENT, "x and y must be 16-byte aligned");
  const int64_t kred = (int64_t)C * R * S;
  r = check_weights(w, K, kred);
  if (r != DS_OK) return r;
  r = check_image(C, H, W, OH, OW);
  if (r != DS_OK) return r;
  const int64_t xb = int32_tensor_bytes({N, C, H, W}), yb = int32_tensor_bytes({N, K, OH, OW});
  if (xb < 0 || yb < 0) return fail(DS_ERR_UNSUPPORTED, "x or y larger than 2^62 bytes");
  if (ranges_overlap(x, xb, y, yb)) return fail(DS_ERR_INVALID_ARG, "y must not overlap x");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  GemmParams p{};
  p.x = x;
  p.bias = bias;
  p.residual = (flags & DS_RESIDUAL) ? residual : nullptr;
  p.y = y;
  p.rows = (int64_t)N * OH * OW;
  p.kred = kred;
  p.cols = K;
  p.flags = flags;
  p.C = C;
  p.H = H;
  p.W = W;
  p.R = R;
  p.S = S;
  p.sh = stride_h;
  p.sw = stride_w;
  p.ph = pad_h;
  p.pw = pad_w;
  p.OH = OH;
  p.OW = OW;
  fill_blob_offsets(p, w);
  r = prepare_amax(x, xb / (int64_t)sizeof(int32_t), flags, amax_io, st, p);
  if (r != DS_OK) return r;
  if (!(flags & DS_CONV_IM2COL)) {
    if (conv_pointwise_supported(p))
      return cuda_check(launch_conv2d_pointwise(p, st), "conv2d_shift (pointwise) launch");
    if (conv_direct_supported(p)) return cuda_check(launch_conv2d_direct(p, st), "conv2d_shift (direct) launch");
  }
  return cuda_check(launch_conv2d_shift(p, st), "conv2d_shift (implicit GEMM) launch");
}

}  // extern "C"

extern "C" {

ds_status ds_specialize_conv2d_shift(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride,
                                     int pad, ds_specialized** out) {
  NvtxRange nvtx_range("ds_specialize_conv2d_shift");
  clear_error();
  if (!s || !p || !out) return fail(DS_ERR_INVALID_ARG, "NULL pointer argument");
  *out = nullptr;
  if (K <= 0 || C <= 0 || R <= 0 || S <= 0) return fail(DS_ERR_SHAPE, "K, C, R and S must be positive");
  if (stride < 1 || stride > 2 || pad < 0 || pad >= R || pad >= S || R > 11 || S > 11)
    return fail(DS_ERR_UNSUPPORTED, "specialisation supports strides 1 and 2, kernels up to 11, pads below the kernel");
  const int64_t n = (int64_t)K * C * R * S;
  if (n > DS_SPECIALIZE_MAX_WEIGHTS)
    return fail(DS_ERR_UNSUPPORTED, "%lld weights: specialisation holds at most %d", (long long)n,
                DS_SPECIALIZE_MAX_WEIGHTS);
  for (int64_t i = 0; i < n; ++i)
    if (s[i] < -1 || s[i] > 1 || p[i] < -15 || p[i] > 0)
      return fail(DS_ERR_CODE_RANGE, "code %lld out of range (s = %d, p = %d)", (long long)i, s[i], p[i]);
  return specialize_conv(s, p, K, C, R, S, stride, pad, out);
}

ds_status ds_conv2d_shift_specialized(const ds_specialized* h, const int32_t* x, const int32_t* bias,
                                      const int32_t* residual, int32_t* y, int N, int H, int W, uint32_t flags,
                                      uint32_t* amax_io, void* stream) {
  NvtxRange nvtx_range("ds_conv2d_shift_specialized");
  clear_error();
  if (!h) return fail(DS_ERR_INVALID_ARG, "NULL specialised layer");
  if (!x || !y) return fail(DS_ERR_INVALID_ARG, "NULL x or y");
  if (N <= 0) return fail(DS_ERR_SHAPE, "N must be positive");
  int K = 0, C = 0, R = 0, S = 0, stride = 0, pad = 0;
  specialized_dims(h, &K, &C, &R, &S, &stride, &pad);
  int OH = 0, OW = 0;
  ds_status r = window_output(H, W, R, S, stride, stride, pad, pad, &OH, &OW);
  if (r != DS_OK) return r;
  const uint32_t known = DS_RELU | DS_AMAX_IN | DS_AMAX_OUT | DS_RESIDUAL | DS_FORCE_INT64;
  if (flags & ~known) return fail(DS_ERR_INVALID_ARG, "unknown flag bits 0x%x", flags & ~known);
  if ((flags & DS_RESIDUAL) && residual == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_RESIDUAL needs a residual tensor");
  if ((flags & (DS_AMAX_IN | DS_AMAX_OUT)) && amax_io == nullptr)
    return fail(DS_ERR_INVALID_ARG, "DS_AMAX_IN / DS_AMAX_OUT need amax_io");
  if (!aligned16(x) || !aligned16(y)) return fail(DS_ERR_ALIGNMENT, "x and y must be 16-byte aligned");
  r = check_image(C, H, W, OH, OW);
  if (r != DS_OK) return r;
  const int64_t xb = int32_tensor_bytes({N, C, H, W}), yb = int32_tensor_bytes({N, K, OH, OW});
  if (xb < 0 || yb < 0) return fail(DS_ERR_UNSUPPORTED, "x or y larger than 2^62 bytes");
  if (ranges_overlap(x, xb, y, yb)) return fail(DS_ERR_INVALID_ARG, "y must not overlap x");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  GemmParams p{};
  p.flags = flags;
  r = prepare_amax(x, xb / (int64_t)sizeof(int32_t), flags, amax_io, st, p);
  if (r != DS_OK) return r;
  return cuda_check(launch_specialized(h, x, bias, (flags & DS_RESIDUAL) ? residual : nullptr, y, N, H, W, OH, OW,
                                       flags, (flags & DS_FORCE_INT64) ? nullptr : p.amax_in, p.amax_out, st),
                    "specialised conv2d_shift launch");
}

void ds_specialized_destroy(ds_specialized* h) { destroy_specialized(h); }

}  // extern "C"

