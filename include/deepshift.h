/*
 * deepshift.h -- C ABI of the DeepShift shift-operator library for GB300 (sm_103a).
 *
 * DeepShift (Elhoushi et al., "DeepShift: Towards Multiplication-Less Neural
 * Networks") replaces every multiply of a fully-connected or convolutional
 * layer by a bitwise shift and a sign flip (Sec. 3, Eq. 1-3).  With weight
 * codes s in {-1, 0, +1} (Eq. 2) and p in [-15, 0] (Sec. 4) and int32
 * activations / biases in 32-bit fixed point with 16 fraction bits (Sec. 4),
 * every operator of this library computes, per output,
 *
 *     y = ReLU?( sat32( b + sum_k s_k * (x_k >> -p_k) ) )
 *
 * with ">>" the two's-complement arithmetic right shift (floor division by
 * 2^-p, Eq. 1), the shift applied before the flip, the sum exact and the
 * result saturated to the int32 range.
 *
 * Conventions for every entry point:
 *   - Tensor pointers are DEVICE pointers owned by the caller.  The library
 *     allocates no memory in any call.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Compute calls are asynchronous and stream-ordered; only
 *     ds_pack_shift_weights synchronises its stream.
 *   - Arguments are validated before anything is launched.  On an error the
 *     call returns a non-zero ds_status, launches nothing, writes no output,
 *     and ds_last_error() describes the problem.  A failed launch returns
 *     DS_ERR_CUDA.
 *   - Activation / output base pointers must be 16-byte aligned
 *     (DS_ERR_ALIGNMENT otherwise).  Any positive size is accepted; tails are
 *     handled inside the kernels.
 */
#ifndef DEEPSHIFT_H
#define DEEPSHIFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DS_OK = 0,
  DS_ERR_INVALID_ARG = 1,      /* null pointer, bad flag, inconsistent descriptor */
  DS_ERR_SHAPE = 2,            /* non-positive or inconsistent dimension */
  DS_ERR_CODE_RANGE = 3,       /* s not in {-1,0,1} or p not in [-15,0] */
  DS_ERR_ALIGNMENT = 4,        /* pointer not 16-byte aligned */
  DS_ERR_BUFFER_TOO_SMALL = 5, /* caller buffer smaller than required */
  DS_ERR_UNSUPPORTED = 6,      /* valid but not supported (e.g. too large) */
  DS_ERR_CUDA = 7              /* a CUDA runtime call or launch failed */
} ds_status;

/* Devices.  Kernel attributes (the opt-in shared-memory size, non-portable
 * cluster sizes) are set once per process, on the device that is current at a
 * kernel's first launch: drive one GPU per process (one process per GPU, as
 * the multi-GPU replicas do).  A launch on a second device from the same
 * process is not supported; it fails with DS_ERR_CUDA rather than computing
 * anything wrong.  The device's SM count, which sizes grids, split
 * reductions and cluster choices, is likewise read once per process. */

/* Size limits.  Every size the library forms from caller dimensions is
 * bounded before it can overflow 64 bits.  A code matrix holds at most 2^48
 * codes, with n_out <= 2^31 and k_red <= 2^40 (2^36 for the expanded and
 * bf16 layouts); a tensor holds at most 2^62 bytes; a zero-padded image
 * extent (H + 2 pad) is at most 2^31 - 1; one convolution image has at most
 * 2^31 input values (C x H x W) and 2^30 output positions (OH x OW).  Larger
 * dimensions give DS_ERR_UNSUPPORTED, and 0 from the size queries. */

/* Description of the last error on the calling thread ("" if none). */
const char* ds_last_error(void);

/* Library version: major * 10000 + minor * 100 + patch (a library utility: no counterpart in the paper). */
int ds_version(void);

/* sizeof of the ABI structs as compiled into the library (0: ds_weights, 1: ds_layer), so that
 * bindings can check their layout; 0 for any other argument (a library utility: no counterpart in the paper). */
size_t ds_abi_struct_size(int which);

/* ---------------------------------------------------------------------------
 * Flags of the compute calls
 * ------------------------------------------------------------------------- */
#define DS_RELU 1u      /* y = max(y, 0) after saturation (and after the residual add) */
#define DS_AMAX_IN 2u   /* amax_io[0] already holds max|x| of the input: skip the pre-pass */
#define DS_AMAX_OUT 4u  /* write max|y| over this call's outputs into amax_io[1] */
#define DS_RESIDUAL 8u  /* conv only: y = sat32(sat32(conv) + residual) before the ReLU */
#define DS_FORCE_INT64 16u /* always use the 64-bit accumulator path (testing / worst case) */
#define DS_CONV_IM2COL 32u /* conv only: use the implicit-GEMM (im2col gather) kernel instead of the
                              direct halo-tile kernel (testing / comparison) */

/* ---------------------------------------------------------------------------
 * Packed weights.
 *
 * A layer's codes are given as two int8 matrices s[n_out][k_red] and
 * p[n_out][k_red], row-major (a conv layer's OIHW codes flattened, so
 * k_red = C*R*S in (c, r, s) order).  They are packed once into a blob of
 * ds_packed_weight_bytes(n_out, k_red) bytes in caller-owned device memory.
 *
 * Blob layout (format DS_FORMAT_PLANES6, all offsets in bytes, little endian):
 *   [0, 256)          header written by the pack kernel:
 *                       u32 magic (0x31575344 "DSW1"), u32 format,
 *                       i64 n_out, i64 k_red, i64 n_chunks,
 *                       u32 invalid_count, u32 nnz_max, u64 a_max
 *   nib  @ 256        n_chunks x n_out records of 4 u32: for chunk g, column n,
 *                     word w holds in bits 4i..4i+3 the value -p (0..15) of
 *                     reduction index k = 32g + 8w + i
 *   bits @ nib + n_chunks*n_out*16
 *                     n_chunks x n_out records of 2 u32 {sign, nz}: bit j of
 *                     `sign` is set iff s = -1 and bit j of `nz` iff s != 0,
 *                     for k = 32g + j
 *   colA @ bits + n_chunks*n_out*8
 *                     n_out u64: A[n] = sum_k |s| * 2^(15 + p)  (sum of |w| in
 *                     units of 2^-15; used to prove int32 accumulation exact)
 *   nnz  @ colA + n_out*8
 *                     n_out u32: number of non-zero codes of column n
 * Entries with k >= k_red are zero codes.  n_chunks = ceil(k_red / 32).
 * Storage is 6 bits per weight: 4 shift bits + sign + non-zero.  The paper's
 * 5-bit count (Sec. 4) has 32 states, one short of the 33 states of a ternary
 * sign times 16 shifts, so the non-zero plane is the sixth bit (layers whose
 * shifts stay in [-14, 0] can be stored in 5 bits: DS_FORMAT_CODES5 below).
 * ------------------------------------------------------------------------- */
#define DS_FORMAT_PLANES6 1u
#define DS_WEIGHTS_MAGIC 0x31575344u

typedef struct ds_weights {
  uint32_t magic;       /* DS_WEIGHTS_MAGIC once filled by ds_pack_shift_weights */
  uint32_t format;      /* DS_FORMAT_PLANES6 */
  int64_t n_out;        /* output columns (FC: N, conv: K) */
  int64_t k_red;        /* reduction length (FC: K, conv: C*R*S) */
  int64_t n_chunks;     /* ceil(k_red / 32) */
  const void* packed;   /* device pointer to the blob (caller-owned, must outlive use) */
  size_t packed_bytes;  /* size of the blob */
  uint64_t a_max;       /* max over columns of A[n] */
  uint32_t nnz_max;     /* max over columns of the non-zero count */
  uint32_t reserved;
  const void* expanded; /* NULL, or the execution layout set by ds_expand_shift_weights */
  size_t expanded_bytes;
  const void* weights_bf16; /* NULL, or the bf16 weights set by ds_expand_shift_weights_bf16 */
  size_t weights_bf16_bytes;
} ds_weights;

/* Bytes needed for the packed blob of an n_out x k_red code matrix (0 if invalid). */
size_t ds_packed_weight_bytes(int64_t n_out, int64_t k_red);

/*
 * Pack codes (Eq. 3's shift matrix P and sign matrix S, Sec. 4 range).
 *   s, p       device int8 [n_out][k_red], row-major.
 *   packed     device buffer of at least ds_packed_weight_bytes(n_out, k_red)
 *              bytes, 256-byte aligned (cudaMalloc / torch allocations are).
 *   desc       host struct filled on success.
 * Synchronises `stream` (an offline call) so that it can report
 * DS_ERR_CODE_RANGE when any s is outside {-1,0,1} or p outside [-15,0]
 * (the blob is then unusable and desc is not filled).
 */
ds_status ds_pack_shift_weights(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red,
                                void* packed, size_t packed_bytes, ds_weights* desc, void* stream);

/* ---------------------------------------------------------------------------
 * Strict 5-bit code storage (Sec. 4: 4 shift bits and a sign bit per weight).
 *
 * With every shift of a nonzero weight in [-14, 0], a ternary sign times 15
 * shifts plus the zero weight is 31 states, which fit 5 bits: code 0 is the
 * zero weight, 1 + (-p) a weight with s = +1, 16 + (-p) one with s = -1 (31
 * is never written).  This is a storage format for such layers: compute calls
 * take the 6-bit blob above, made from the codes that ds_unpack_shift_weights5
 * returns.  The p of a zero weight is not stored and reads back as 0 (no term
 * depends on it).
 *
 * Blob layout (format DS_FORMAT_CODES5, little endian):
 *   [0, 256)     header: u32 magic (0x31575344), u32 format (2), i64 n_out,
 *                i64 k_red, i64 n_chunks = ceil(k_red / 32), u32 invalid_count
 *   @ 256        n_out x n_chunks records of 5 u32, record (n, g) at
 *                256 + 20 (n n_chunks + g): bit j of word b is bit b of the
 *                code of k = 32 g + j (zero beyond k_red)
 * 5 bits per weight, the total rounded up to 256 bytes.
 * ------------------------------------------------------------------------- */
#define DS_FORMAT_CODES5 2u

/* Bytes of the 5-bit blob of an n_out x k_red code matrix (0 if invalid). */
size_t ds_packed5_weight_bytes(int64_t n_out, int64_t k_red);

/*
 * Store codes (s, p: device int8 [n_out][k_red], row-major) in the 5-bit blob
 * `packed5` (device, 256-byte aligned, at least ds_packed5_weight_bytes bytes,
 * caller-owned).  Synchronises `stream` (an offline call) so that it can
 * report DS_ERR_CODE_RANGE when a code has no 5-bit state (s outside
 * {-1, 0, 1}, or p outside [-14, 0] for s != 0, or outside [-15, 0] for s = 0);
 * the blob is then unusable.
 */
ds_status ds_pack_shift_weights5(const int8_t* s, const int8_t* p, int64_t n_out, int64_t k_red, void* packed5,
                                 size_t packed5_bytes, void* stream);

/*
 * Read a 5-bit blob back into s, p (device int8 [n_out][k_red], caller-owned;
 * p = 0 where s = 0).  Synchronises `stream`: the header is checked on the
 * host first (DS_ERR_INVALID_ARG: not a 5-bit blob; DS_ERR_SHAPE: other
 * dims), and DS_ERR_CODE_RANGE reports codes 31 (written as zero weights).
 */
ds_status ds_unpack_shift_weights5(const void* packed5, size_t packed5_bytes, int64_t n_out, int64_t k_red,
                                   int8_t* s, int8_t* p, void* stream);

/* ---------------------------------------------------------------------------
 * Expanded execution layout (optional).  The packed blob is the storage
 * format; decoding it inside every CTA of every launch costs a measurable
 * share of the integer issue slots of these ALU-bound kernels.  A layer may
 * therefore be expanded once into 32-bit shift / sign words laid out as the
 * kernels stage them:
 *   int32 [ceil(n_out / 32)][k_red][64]: for column block cb and reduction
 *   index k, words 0..31 hold -p and words 32..63 hold s of columns
 *   32*cb .. 32*cb + 31 (zero beyond n_out).
 * 8 bytes per weight (plus padding of the last column block).  Kernels use
 * it when desc->expanded is set and decode the blob otherwise; results are
 * identical either way.
 * ------------------------------------------------------------------------- */

/* Bytes of the expanded layout of an n_out x k_red code matrix (0 if invalid). */
size_t ds_expanded_weight_bytes(int64_t n_out, int64_t k_red);

/*
 * Expand packed weights (the codes of Eq. 3's flip(2^P, S)) into `expanded` (device, 16-byte aligned, at least
 * ds_expanded_weight_bytes bytes, caller-owned and outliving every use) and
 * record it in *w (w->expanded, w->expanded_bytes).  Stream-ordered and
 * asynchronous; the blob must stay valid.  Errors: DS_ERR_INVALID_ARG for an
 * unfilled descriptor, DS_ERR_BUFFER_TOO_SMALL, DS_ERR_ALIGNMENT.
 */
ds_status ds_expand_shift_weights(ds_weights* w, void* expanded, size_t expanded_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Float variant (bf16 activations, fp32 accumulation on the tensor cores).
 *
 * With x in bf16 the product x * s * 2^p is exact (s * 2^p is a power of two
 * with p in [-15, 0]), so LinearShift is an ordinary dense contraction
 *     y[m][n] = ReLU?( bias[n] + sum_k x[m][k] * W[n][k] ),  W = flip(2^P, S)  (Eq. 3)
 * with fp32 accumulation.  Its result is not bit-exact: the sum is rounded
 * in an implementation-defined order; |y - exact| <= 1e-5 * (sum_k |x W| + |bias|)
 * is the tolerance the tests hold it to.
 * ------------------------------------------------------------------------- */

/* Bytes of the bf16 weight layout: bf16 [n_out][kpad], kpad = ceil(k_red / 8) * 8. */
size_t ds_bf16_weight_bytes(int64_t n_out, int64_t k_red);

/*
 * Decode packed weights into bf16 W[n][k] = s * 2^p = flip(2^P, S) of Eq. 3 (sign bit, exponent 127 + p,
 * zero mantissa; +0 for s = 0) in `buf` (device, 16-byte aligned, caller-owned)
 * and record it in w->weights_bf16.  Stream-ordered, asynchronous.
 */
ds_status ds_expand_shift_weights_bf16(ds_weights* w, void* buf, size_t bytes, void* stream);

/*
 * Float LinearShift (Eq. 3, fully-connected form, in the float form the paper trains with, Sec. 4) on tcgen05
 * tensor cores (TMA-fed, TMEM accumulator).
 *   x     device bf16 bit patterns (uint16) [M][K], row-major, K % 8 == 0
 *   w     weights with w->weights_bf16 set, n_out == N, k_red == K
 *   bias  device fp32 [N] or NULL
 *   y     device fp32 [M][N]
 *   flags DS_RELU or 0
 * Errors: DS_ERR_UNSUPPORTED when K % 8 != 0 or the bf16 weights are missing.
 */
ds_status ds_linear_shift_bf16(const uint16_t* x, const ds_weights* w, const float* bias, float* y, int64_t M,
                               int64_t K, int64_t N, uint32_t flags, void* stream);

/* 1 if a bounded wait of the float kernel gave up in any ds_linear_shift_bf16 launch since the previous call of
 * this function (or since the library loaded), 0 if none did, -1 if the flag could not be read.  Reading clears
 * the flag.  The flag is device-wide and not per call: synchronise the streams of the calls it should cover
 * first (the read itself is a synchronous copy).  A launch whose wait gave up stops early, so its y is
 * incomplete.  A library utility: no counterpart in the paper. */
int ds_bf16_fault_flag(void);

/* Diagnostic: the limit, in SM clock cycles, of each bounded wait of the float kernel's later launches; cycles <= 0
 * restores the default (4e9 cycles, about 2 s).  A launch whose wait runs out stops issuing work, lets the copies and
 * tensor-core operations it already issued finish, frees its tensor memory and sets the fault flag above, so a test
 * can make the waits run out on purpose and the context stays usable.  Process-wide (not per stream or thread).
 * A library utility: no counterpart in the paper. */
void ds_bf16_set_wait_limit(long long cycles);

/* ---------------------------------------------------------------------------
 * Accumulator width.  Each compute call proves, on the device and with no
 * host round trip, whether 32-bit accumulation is exact:
 *     ceil(amax * A[n] / 2^15) + nnz[n] + |b[n]| <= 2^31 - 1   for every n
 * where amax = max|x| of the input.  If so the 32-bit path runs (no
 * wrap-around and no saturation can occur); otherwise a 64-bit path runs and
 * the exact sum is saturated.  amax comes from amax_io[0] when DS_AMAX_IN is
 * set, else from a pre-pass over x that writes it to amax_io[0].  amax_io
 * (device, 2 x u32) may be NULL: then no bound is available and the 64-bit
 * path is always taken (DS_AMAX_IN and DS_AMAX_OUT need amax_io).
 * ------------------------------------------------------------------------- */

/*
 * LinearShift forward (Eq. 3, Y = flip(2^P, S) X + b; Sec. 4 fixed point):
 *   y[m][n] = sat32( bias[n] + sum_k s[n][k] * (x[m][k] >> -p[n][k]) ), ReLU if DS_RELU.
 *   x     device int32 [M][K] row-major (Q16.16)
 *   w     packed weights with n_out == N and k_red == K
 *   bias  device int32 [N] or NULL (zero bias)
 *   y     device int32 [M][N] row-major; must not overlap x
 *   amax_io device u32[2] or NULL (see above); DS_AMAX_OUT writes max|y| to amax_io[1]
 */
ds_status ds_linear_shift(const int32_t* x, const ds_weights* w, const int32_t* bias, int32_t* y,
                          int64_t M, int64_t K, int64_t N, uint32_t flags, uint32_t* amax_io,
                          void* stream);

/*
 * ConvShift forward (Eq. 3, Y = flip(2^P, S) (*) X + b; cross-correlation with
 * zero padding, as the paper's PyTorch operator):
 *   y[n][k][oh][ow] = sat32( bias[k] + sum_{c,r,q} s[k][c][r][q] *
 *                            (xpad[n][c][oh*sh + r][ow*sw + q] >> -p[k][c][r][q]) )
 *   then, with DS_RESIDUAL, y = sat32(y + residual[n][k][oh][ow]); then ReLU if DS_RELU.
 *   x        device int32 NCHW [N][C][H][W]
 *   w        packed weights with n_out == K and k_red == C*R*S
 *   bias     device int32 [K] or NULL
 *   residual device int32 NCHW [N][K][OH][OW], required iff DS_RESIDUAL
 *   y        device int32 NCHW [N][K][OH][OW], OH = (H + 2*pad_h - R)/stride_h + 1
 *   amax_io  as for ds_linear_shift
 */
ds_status ds_conv2d_shift(const int32_t* x, const ds_weights* w, const int32_t* bias,
                          const int32_t* residual, int32_t* y, int N, int C, int H, int W, int K,
                          int R, int S, int stride_h, int stride_w, int pad_h, int pad_w,
                          uint32_t flags, uint32_t* amax_io, void* stream);

/*
 * LinearShift for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment convenience of this library.
 *
 * Same operation, arguments and errors as ds_linear_shift, except that the
 * two scratch words of amax_io come from a static device array of 64 u32
 * (256 bytes) that every GPU loading this library holds until the process
 * exits.  It suits callers that must not call cudaMalloc or any allocating
 * routine: a plugin given only its input and output buffers, a host callback,
 * a real-time path that must stay out of the allocator.  Each call uses two of
 * the 64 words whatever the problem size; a build whose per-call need exceeded
 * the array would be rejected with DS_ERR_UNSUPPORTED.  DS_AMAX_IN and
 * DS_AMAX_OUT are rejected (DS_ERR_INVALID_ARG): they need caller scratch.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress with that device current) and caches it; make that
 *     first call before any stream capture.
 *   - All calls share the array, which keeps the last call's contents; the
 *     max|x| pre-pass clears its word before writing it.  Calls that overlap on
 *     the GPU (different streams without ordering, or several threads) race on
 *     the array and may compute wrong results: order them on one stream.
 *   - It allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 */
ds_status ds_linear_shift_static_scratch(const int32_t* x, const ds_weights* w, const int32_t* bias,
                                         int32_t* y, int64_t M, int64_t K, int64_t N, uint32_t flags,
                                         void* stream);

/* ---------------------------------------------------------------------------
 * Chained forward (ResNet / VGG shaped networks of shift layers).
 *
 * A network is an array of ds_layer run in program order.  Tensors
 * live in numbered slots: slot 0 is the network input x, slot 1 the network
 * output y, slots >= 2 are carved from the caller's workspace.  Activations
 * are NCHW int32 Q16.16; an FC layer reads its input slot as [batch][C*H*W].
 * The ops are the paper's operators (Eq. 3: DS_OP_CONV, DS_OP_FC with the
 * fused bias / saturation / residual / ReLU epilogue) plus the integer pools
 * that ResNet and VGG need (DS_OP_MAXPOOL: max over the window, padded taps
 * ignored; DS_OP_AVGPOOL: floor(sum / (R*S)), no padding).  Each shift layer
 * proves its accumulator width on the device from the max|x| that its
 * producer wrote (the network input gets one pre-pass), so the whole forward
 * runs without a host round trip and can be captured in a CUDA graph.  Make one
 * eager call with the same program and batch first: the first launch of each
 * kernel shape sets kernel attributes and queries cluster occupancy, host calls
 * that a capture in the default (global) mode may refuse.
 * ------------------------------------------------------------------------- */
#define DS_OP_CONV 1
#define DS_OP_FC 2
#define DS_OP_MAXPOOL 3
#define DS_OP_AVGPOOL 4

typedef struct ds_layer {
  int32_t op;          /* DS_OP_* */
  int32_t in;          /* input slot */
  int32_t aux;         /* residual slot (DS_RESIDUAL), else -1 */
  int32_t out;         /* output slot (not 0; distinct from in and aux) */
  int32_t C, H, W;     /* input channels and spatial size, per image */
  int32_t K;           /* conv / FC: output channels or features (pools: ignored) */
  int32_t R, S;        /* conv / pool window */
  int32_t stride, pad; /* conv / pool */
  uint32_t flags;      /* DS_RELU, DS_RESIDUAL (conv only) */
  const ds_weights* w; /* conv / FC weights (n_out = K, k_red = C*R*S or C*H*W) */
  const int32_t* bias; /* conv / FC bias (device int32 [K]) or NULL */
} ds_layer;

/*
 * Workspace bytes for running n layers at the given batch (0 if invalid):
 * every slot >= 2 sized for the largest tensor written to it, plus the
 * max|x| words.  Validates the program like ds_shift_forward.
 */
size_t ds_shift_forward_workspace_bytes(const ds_layer* layers, int n, int batch);

/*
 * Runs the program (shift layers of Eq. 3 with the Sec. 4 fixed point, pools as described above):
 * x = slot 0 (device, [batch][C0][H0][W0] of layer 0),
 * y = slot 1 (device, the tensor of the last layer that writes slot 1),
 * ws = workspace (device, 256-byte aligned, >= the bytes above).
 * Validation errors (DS_ERR_SHAPE, DS_ERR_INVALID_ARG, ...) are reported
 * before anything is launched.  Asynchronous, stream-ordered, no device
 * allocation; the planner's small host arrays are allocated before the first
 * launch, and a failed host allocation returns DS_ERR_UNSUPPORTED ("host
 * memory allocation failed") with nothing launched.  No C++ exception leaves
 * any entry point.
 * A layer that depends on neither its predecessor's output nor a slot that
 * its predecessor reads or writes (a ResNet block's shortcut beside the main
 * branch) runs on a side stream of the calling thread, ordered by events on
 * the slots it reads and writes; the caller's stream waits for the side
 * stream before the call returns, so `stream` orders everything as before.
 * The side stream and its events are created on a thread's first call (one
 * set per host thread, kept until the thread ends); if they cannot be
 * created, every layer runs on `stream`.
 */
ds_status ds_shift_forward(const ds_layer* layers, int n, const int32_t* x, int32_t* y, void* ws,
                           size_t ws_bytes, int batch, void* stream);

/* ---------------------------------------------------------------------------
 * Input gradient (Eq. 7 and its footnote: dC/dX = dC/dY W_q^T for LinearShift,
 * W_q^rot180 (*) dC/dY for ConvShift).  The gradient dY is int32 Q16.16 and
 * each term is the forward's shift-then-flip, s * (dy >> -p); the exact sum
 * is saturated to int32 (no bias, no ReLU).
 *
 * ds_pack_shift_weights_backward packs the code matrices of that pass from
 * the forward codes s, p (device int8, [K][C][R][S]; an FC layer's [N][K_in]
 * is K = N, C = K_in, R = S = 1, strides 1).  A layer of strides (sh, sw) has
 * sh * sw tap phases (a, b): input position i = sh i' + rho receives only the
 * taps r = a + sh t with a = (rho + pad) mod sh, so each phase is a stride-1
 * correlation of dY with a sub-kernel of Th(a) = ceil((R - a) / sh) x Tw(b)
 * taps.  Phase (a, b) is packed as a matrix of C columns and reduction length
 * K * Th * Tw (index (k, t, u) holds the code of (k, c, a + sh (Th-1-t),
 * b + sw (Tw-1-u)); for stride 1 this is W^rot180 with the channels swapped)
 * into desc[a * sw + b]; a phase with no taps gets a descriptor with
 * k_red = 0 and no blob.  desc points to sh * sw caller-owned descriptors,
 * packed to ds_packed_weight_bytes_backward(K, C, R, S, sh, sw) bytes
 * (256-byte aligned; phases at 256-byte aligned offsets).  Synchronises its
 * stream once per phase; DS_ERR_CODE_RANGE on bad codes; strides in [1, 16].
 *
 * ds_linear_shift_backward_x: dx [M][K] from dy [M][N] (row-major, 16-byte
 * aligned) with w_bwd packed by ds_pack_shift_weights_backward(s, p, N, K,
 * 1, 1, 1, 1, ...).  Flags: DS_AMAX_IN / DS_AMAX_OUT (amax_io as in
 * ds_linear_shift) and DS_FORCE_INT64 only.
 *
 * ds_conv2d_shift_backward_x: dx [N][C][H][W] from dy [N][K][OH][OW] of the
 * forward geometry (H, W, R, S, strides, pads as given to ds_conv2d_shift;
 * OH = (H + 2 pad_h - R) / stride_h + 1, likewise OW), w_bwd the
 * stride_h * stride_w descriptors of ds_pack_shift_weights_backward(s, p, K,
 * C, R, S, stride_h, stride_w, ...).  Stride 1 runs the forward ConvShift of
 * dy with padding R-1-pad (direct / pointwise kernels); larger strides run one
 * implicit GEMM per output phase (no term of a skipped window position is
 * computed) and zero-fill the positions no tap reaches.  Flags: DS_AMAX_IN,
 * DS_AMAX_OUT, DS_FORCE_INT64, and DS_CONV_IM2COL (the per-phase implicit
 * GEMM also at stride 1).  Errors as ds_conv2d_shift.
 * ------------------------------------------------------------------------- */
size_t ds_packed_weight_bytes_backward(int K, int C, int R, int S, int stride_h, int stride_w);
ds_status ds_pack_shift_weights_backward(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride_h,
                                         int stride_w, void* packed, size_t packed_bytes, ds_weights* desc,
                                         void* stream);
ds_status ds_linear_shift_backward_x(const int32_t* dy, const ds_weights* w_bwd, int32_t* dx, int64_t M, int64_t K,
                                     int64_t N, uint32_t flags, uint32_t* amax_io, void* stream);
ds_status ds_conv2d_shift_backward_x(const int32_t* dy, const ds_weights* w_bwd, int32_t* dx, int N, int C, int H,
                                     int W, int K, int R, int S, int stride_h, int stride_w, int pad_h, int pad_w,
                                     uint32_t flags, uint32_t* amax_io, void* stream);

/* ---------------------------------------------------------------------------
 * Conversion of float models (the step before packing).
 *
 * ds_quantize_shift_weights: the DeepShift-Q quantizer (Sec. 3.1, Eq. 4-6,
 * with the shift clipping of Sec. 4) of n float32 weights w (device, 4-byte
 * aligned, any layout; conv weights flattened as [K][C][R][S]) into the
 * int8 codes s (device, n bytes) and p (device, n bytes) that
 * ds_pack_shift_weights takes:
 *   s = sign(w) in {-1, 0, +1},  p = clip(round(log2|w|), p_min, 0).
 * round(log2|w|) is the integer n with 2^(n-1/2) <= |w| < 2^(n+1/2), decided
 * exactly (no float log; no float weight is a tie).  p_min is -15 (the
 * 6-bit code format) or -14 (codes that also fit the strict 5-bit format of
 * Sec. 4); other values in [-15, 0] are accepted.  w = 0 and NaN give s = 0,
 * p = p_min; +-inf gives s = +-1, p = 0.  Stream-ordered, no synchronisation.
 * Errors: DS_ERR_INVALID_ARG (NULL pointer, p_min outside [-15, 0]),
 * DS_ERR_SHAPE (n <= 0), DS_ERR_ALIGNMENT (w not 4-byte aligned).
 *
 * ds_quantize_q16: Sec. 4's rounding of float inputs (and biases) to 32-bit
 * fixed point with 16 fraction bits: q = round-half-to-even(x * 2^16),
 * saturated to [INT32_MIN, INT32_MAX]; NaN gives 0.  x (n float32) and q
 * (n int32) are device pointers, 4-byte aligned (16-byte alignment takes
 * the vectorised path).  Errors: DS_ERR_INVALID_ARG, DS_ERR_SHAPE,
 * DS_ERR_ALIGNMENT as above.
 * ------------------------------------------------------------------------- */
ds_status ds_quantize_shift_weights(const float* w, int64_t n, int p_min, int8_t* s, int8_t* p, void* stream);
ds_status ds_quantize_q16(const float* x, int64_t n, int32_t* q, void* stream);

/*
 * max |x| over n int32 values, written to *amax (device u32; |INT32_MIN| = 2^31): the input of the
 * accumulator-width proof above (the paper is silent on overflow; Sec. 4 fixes only the 32-bit format).
 */
ds_status ds_absmax(const int32_t* x, int64_t n, uint32_t* amax, void* stream);

/* ---------------------------------------------------------------------------
 * Weight-specialised ConvShift (Eq. 3, as ds_conv2d_shift; specialising the kernels to the weights at run time is
 * the future work of Sec. 6.1).  For a small layer the library writes a kernel in which every weight's shift and
 * sign are immediates and the zero weights are left out, so a term is one shift by an immediate and one add or
 * subtract (no shift for p = 0), with no code loads; it compiles the kernel at run time with NVRTC (libnvrtc,
 * opened on first use) for the current device and keeps it in the returned handle.  Meant for the few-thousand-
 * weight layers at the input of a network (VGG16's first conv: 1728 weights), where the whole layer fits the
 * instruction stream.
 *
 * ds_specialize_conv2d_shift: s, p HOST int8 codes [K][C][R][S] (s in {-1, 0, +1}, p in [-15, 0]); square
 * stride (1 or 2) and padding (below R and S); K*C*R*S <= DS_SPECIALIZE_MAX_WEIGHTS, R, S <= 11.  Compiles and
 * loads (seconds for the largest layers; not stream-ordered, not for a capture).  On success *out owns the kernel
 * until ds_specialized_destroy.  Errors: DS_ERR_INVALID_ARG (NULL), DS_ERR_SHAPE, DS_ERR_CODE_RANGE,
 * DS_ERR_UNSUPPORTED (too many weights or channels for the shared-memory tile, NVRTC missing or failing),
 * DS_ERR_CUDA.
 *
 * ds_conv2d_shift_specialized: the layer on x [N][C][H][W] -> y [N][K][OH][OW] (NCHW int32, 16-byte aligned,
 * not overlapping), bias, residual, flags (DS_RELU, DS_RESIDUAL, DS_AMAX_IN, DS_AMAX_OUT, DS_FORCE_INT64) and
 * amax_io exactly as ds_conv2d_shift; the same accumulator-width proof picks 32- or 64-bit sums per CTA.  Use it
 * on the device it was specialised on.  Stream-ordered, allocates nothing.
 * ------------------------------------------------------------------------- */
#define DS_SPECIALIZE_MAX_WEIGHTS 4096
typedef struct ds_specialized ds_specialized;
ds_status ds_specialize_conv2d_shift(const int8_t* s, const int8_t* p, int K, int C, int R, int S, int stride,
                                     int pad, ds_specialized** out);
ds_status ds_conv2d_shift_specialized(const ds_specialized* h, const int32_t* x, const int32_t* bias,
                                      const int32_t* residual, int32_t* y, int N, int H, int W, uint32_t flags,
                                      uint32_t* amax_io, void* stream);
void ds_specialized_destroy(ds_specialized* h);

#ifdef __cplusplus
}
#endif

#endif /* DEEPSHIFT_H */
