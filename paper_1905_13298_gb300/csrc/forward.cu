// Chained forward: runs a program of shift layers and integer pools (ResNet /
// VGG shaped networks built from the operators of Eq. 3) on the caller's
// stream, with the layers that do not depend on their predecessor on a side
// stream beside it.
//
// Host side: one validation pass computes every slot's shape, the workspace
// layout, the device max|x| word that bounds each layer's input, and each
// layer's stream and dependencies.  Device side: one memset of the max|x|
// words and split scratch, one max|x| pre-pass over the network input, then
// one launch per layer (plus a finalize for split reductions, and events
// between the streams).  A shift layer reads the max|x| word of
// its producer (pools pass their input's bound through, since max-pool and
// floor-average never exceed it) and writes max|y| into its own word, so the
// accumulator-width proof of every layer happens on the device.
#include <stdio.h>

#include <algorithm>
#include <exception>
#include <vector>

#include "ds_common.cuh"

namespace ds {
namespace {

struct Shape {
  int C = 0, H = 0, W = 0;
  int64_t elems() const { return (int64_t)C * H * W; }
};

struct Plan {
  std::vector<Shape> out_shape;   // per layer
  // two-stream schedule: a layer that does not depend on its predecessor runs on a side stream
  // (a ResNet block's shortcut beside its main branch); deps are the earlier layers (-1: the
  // workspace reset and the input pre-pass) whose results or inputs it must wait for
  std::vector<char> side;
  std::vector<std::vector<int>> deps;
  std::vector<char> signals;      // another stream waits for this layer (index n: the reset)
  bool any_side = false;
  std::vector<int64_t> slot_elems;  // per slot, per image (slots >= 2)
  std::vector<size_t> slot_off;   // byte offsets in the workspace
  size_t amax_bytes = 0;
  size_t split_bytes = 0;  // int64 scratch of split reductions (largest layer)
  size_t total = 0;
  int n_slots = 0;
};

// Re-raises a failed check with the layer's index in front of its message.
ds_status layer_fail(ds_status st, int i) {
  char what[512];
  snprintf(what, sizeof(what), "%s", ds_last_error());
  return fail(st, "layer %d: %s", i, what);
}

// Dependencies through the slots: a layer waits for the last writer of each
// slot it reads (in, aux) and, before it overwrites its output slot, for that
// slot's last writer and every reader since.  A layer that does not depend on
// its predecessor (and whose predecessor runs on the main stream) runs on the
// side stream.
void schedule(const ds_layer* L, int n, Plan& P) {
  std::vector<int> last_writer(P.n_slots, -1);
  std::vector<std::vector<int>> readers(P.n_slots);
  P.side.assign(n, 0);
  P.deps.assign(n, {});
  P.signals.assign(n + 1, 0);
  for (int i = 0; i < n; ++i) {
    const ds_layer& l = L[i];
    std::vector<int>& d = P.deps[i];
    auto add = [&d](int j) {
      if (std::find(d.begin(), d.end(), j) == d.end()) d.push_back(j);
    };
    add(last_writer[l.in]);
    if (l.aux >= 0) add(last_writer[l.aux]);
    add(last_writer[l.out]);
    for (int j : readers[l.out]) add(j);
    P.side[i] = i >= 1 && !P.side[i - 1] && std::find(d.begin(), d.end(), i - 1) == d.end();
    readers[l.in].push_back(i);
    if (l.aux >= 0) readers[l.aux].push_back(i);
    last_writer[l.out] = i;
    readers[l.out].clear();
  }
  for (int i = 0; i < n; ++i) {
    if (P.side[i]) P.any_side = true;
    for (int j : P.deps[i]) {
      const bool j_side = j >= 0 && P.side[j];
      if (j_side != (bool)P.side[i]) P.signals[j >= 0 ? j : n] = 1;
    }
    // a side layer whose dependencies all run on the side stream still waits for the reset of the workspace
    if (P.side[i] && std::none_of(P.deps[i].begin(), P.deps[i].end(), [&](int j) { return j < 0 || !P.side[j]; })) {
      P.deps[i].push_back(-1);
      P.signals[n] = 1;
    }
  }
  // the caller's stream waits for the last side layer before the call returns
  for (int i = n - 1; i >= 0; --i)
    if (P.side[i]) {
      P.signals[i] = 1;
      break;
    }
}

// The side stream and the events of the two-stream schedule, one set per
// host thread (created on first use, kept for the thread's lifetime).
struct SideStream {
  int dev = -1;
  cudaStream_t s = nullptr;
  std::vector<cudaEvent_t> ev;
  SideStream() = default;
  SideStream(const SideStream&) = delete;
  SideStream& operator=(const SideStream&) = delete;
  ~SideStream() { release(); }
  // at thread exit (errors ignored: at process exit the runtime may already be gone)
  void release() {
    for (cudaEvent_t e : ev) (void)cudaEventDestroy(e);
    if (s != nullptr) (void)cudaStreamDestroy(s);
    ev.clear();
    s = nullptr;
    dev = -1;
    (void)cudaGetLastError();
  }
};
thread_local SideStream t_side;

// False when a resource cannot be created: the forward then runs on the caller's stream alone.
bool side_resources(size_t n_events, SideStream*& out) {
  SideStream& S = t_side;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  if (S.dev != dev) {  // a new device for this thread: fresh objects
    S.release();
    if (cudaStreamCreateWithFlags(&S.s, cudaStreamNonBlocking) != cudaSuccess) {
      (void)cudaGetLastError();
      S.s = nullptr;
      return false;
    }
    S.dev = dev;
  }
  while (S.ev.size() < n_events) {
    cudaEvent_t e = nullptr;
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) {
      (void)cudaGetLastError();
      return false;
    }
    S.ev.push_back(e);
  }
  out = &S;
  return true;
}

ds_status plan_program(const ds_layer* L, int n, int batch, Plan& P) {
  if (L == nullptr || n <= 0) return fail(DS_ERR_INVALID_ARG, "empty layer program");
  if (batch <= 0) return fail(DS_ERR_SHAPE, "batch must be positive");
  int max_slot = 1;
  for (int i = 0; i < n; ++i) {
    if (L[i].in < 0 || L[i].out < 1 || L[i].aux < -1)
      return fail(DS_ERR_INVALID_ARG, "layer %d: bad slot numbers", i);
    max_slot = std::max(max_slot, std::max(L[i].in, std::max(L[i].out, L[i].aux)));
  }
  if (max_slot > 64) return fail(DS_ERR_UNSUPPORTED, "at most 64 slots");
  P.n_slots = max_slot + 1;
  std::vector<Shape> slot(P.n_slots);
  std::vector<bool> defined(P.n_slots, false);
  P.slot_elems.assign(P.n_slots, 0);
  P.out_shape.assign(n, Shape{});
  if (L[0].C <= 0 || L[0].H <= 0 || L[0].W <= 0) return fail(DS_ERR_SHAPE, "input image must have positive C, H, W");
  if (check_image(L[0].C, L[0].H, L[0].W, 1, 1) != DS_OK) return fail(DS_ERR_UNSUPPORTED, "input image too large");
  slot[0] = Shape{L[0].C, L[0].H, L[0].W};
  defined[0] = true;
  bool wrote_y = false;
  for (int i = 0; i < n; ++i) {
    const ds_layer& l = L[i];
    if (!defined[l.in]) return fail(DS_ERR_INVALID_ARG, "layer %d reads slot %d before it is written", i, l.in);
    if (l.out == l.in || l.out == l.aux) return fail(DS_ERR_INVALID_ARG, "layer %d: output slot aliases an input", i);
    const Shape in = slot[l.in];
    Shape out;
    switch (l.op) {
      case DS_OP_CONV: {
        if (in.C != l.C || in.H != l.H || in.W != l.W)
          return fail(DS_ERR_SHAPE, "layer %d: input %dx%dx%d, slot holds %dx%dx%d", i, l.C, l.H, l.W, in.C,
                      in.H, in.W);
        if (l.K <= 0 || l.R <= 0 || l.S <= 0 || l.stride <= 0 || l.pad < 0)
          return fail(DS_ERR_SHAPE, "layer %d: bad conv geometry", i);
        int oh = 0, ow = 0;
        ds_status r = window_output(l.H, l.W, l.R, l.S, l.stride, l.stride, l.pad, l.pad, &oh, &ow);
        if (r == DS_OK) r = check_image(l.C, l.H, l.W, oh, ow);
        if (r != DS_OK) return layer_fail(r, i);
        r = check_weights(l.w, l.K, (int64_t)l.C * l.R * l.S);
        if (r != DS_OK) return r;
        out = Shape{l.K, oh, ow};
        P.split_bytes = std::max(P.split_bytes,
                                 conv_split_bytes(conv_params(l.w, batch, l.C, l.H, l.W, l.K, l.R, l.S, l.stride, l.pad)));
        break;
      }
      case DS_OP_FC: {
        if (in.elems() != (int64_t)l.C * l.H * l.W)
          return fail(DS_ERR_SHAPE, "layer %d: FC input of %lld features, slot holds %lld", i,
                      (long long)((int64_t)l.C * l.H * l.W), (long long)in.elems());
        if (l.K <= 0) return fail(DS_ERR_SHAPE, "layer %d: bad FC width", i);
        if (l.K > 65535LL * 64) return fail(DS_ERR_UNSUPPORTED, "layer %d: FC wider than 65535 x 64", i);
        if (l.flags & DS_RESIDUAL) return fail(DS_ERR_INVALID_ARG, "layer %d: residual on FC", i);
        ds_status r = check_weights(l.w, l.K, in.elems());
        if (r != DS_OK) return r;
        out = Shape{l.K, 1, 1};
        break;
      }
      case DS_OP_MAXPOOL:
      case DS_OP_AVGPOOL: {
        if (in.C != l.C || in.H != l.H || in.W != l.W) return fail(DS_ERR_SHAPE, "layer %d: pool input shape", i);
        const int pad = l.op == DS_OP_MAXPOOL ? l.pad : 0;
        if (l.op == DS_OP_AVGPOOL && l.pad != 0) return fail(DS_ERR_UNSUPPORTED, "layer %d: padded avgpool", i);
        if (l.R <= 0 || l.S <= 0 || l.stride <= 0 || pad < 0 || pad >= l.R || pad >= l.S)
          return fail(DS_ERR_SHAPE, "layer %d: bad pool geometry", i);
        int oh = 0, ow = 0;
        ds_status r = window_output(l.H, l.W, l.R, l.S, l.stride, l.stride, pad, pad, &oh, &ow);
        if (r == DS_OK) r = check_image(1, l.H, l.W, oh, ow);  // the pools index one plane at a time
        if (r != DS_OK) return layer_fail(r, i);
        if (l.flags != 0) return fail(DS_ERR_INVALID_ARG, "layer %d: flags on a pool", i);
        out = Shape{l.C, oh, ow};
        break;
      }
      default:
        return fail(DS_ERR_INVALID_ARG, "layer %d: unknown op %d", i, l.op);
    }
    if (l.flags & ~(DS_RELU | DS_RESIDUAL)) return fail(DS_ERR_INVALID_ARG, "layer %d: unsupported flags", i);
    if (l.flags & DS_RESIDUAL) {
      if (l.aux < 0 || !defined[l.aux]) return fail(DS_ERR_INVALID_ARG, "layer %d: residual slot not written", i);
      const Shape a = slot[l.aux];
      if (a.C != out.C || a.H != out.H || a.W != out.W)
        return fail(DS_ERR_SHAPE, "layer %d: residual shape differs from the output", i);
    }
    P.out_shape[i] = out;
    slot[l.out] = out;
    defined[l.out] = true;
    if (l.out == 1) wrote_y = true;
    if (l.out >= 2) P.slot_elems[l.out] = std::max(P.slot_elems[l.out], out.elems());
  }
  if (!wrote_y) return fail(DS_ERR_INVALID_ARG, "no layer writes the output slot 1");
  schedule(L, n, P);
  P.amax_bytes = ((size_t)(n + 1) * sizeof(uint32_t) + 255) / 256 * 256;
  P.split_bytes = (P.split_bytes + 255) / 256 * 256;
  P.slot_off.assign(P.n_slots, 0);
  // the side stream's layers split their reductions in a scratch region of their own
  size_t off = P.amax_bytes + (P.any_side ? 2 : 1) * P.split_bytes;
  for (int s = 2; s < P.n_slots; ++s) {
    P.slot_off[s] = off;
    int64_t bytes = 0;
    if (__builtin_mul_overflow(P.slot_elems[s], (int64_t)batch * (int64_t)sizeof(int32_t), &bytes) ||
        bytes > (int64_t(1) << 62))
      return fail(DS_ERR_UNSUPPORTED, "slot %d larger than 2^62 bytes", s);
    off += ((size_t)bytes + 255) / 256 * 256;
    if (off > (size_t(1) << 62)) return fail(DS_ERR_UNSUPPORTED, "workspace larger than 2^62 bytes");
  }
  P.total = off;
  return DS_OK;
}

}  // namespace
}  // namespace ds

using namespace ds;

extern "C" {

// The planner and the executor keep small host arrays (per slot and per
// layer).  No exception may leave a C entry point: a failed host allocation
// becomes a status, reported before anything is launched (every array exists
// before the first launch).
size_t ds_shift_forward_workspace_bytes(const ds_layer* layers, int n, int batch) {
  clear_error();
  try {
    Plan P;
    if (plan_program(layers, n, batch, P) != DS_OK) return 0;
    return P.total;
  } catch (const std::exception&) {
    fail(DS_ERR_UNSUPPORTED, "host memory allocation failed");
    return 0;
  }
}

static ds_status shift_forward(const ds_layer* L, int n, const int32_t* x, int32_t* y, void* ws, size_t ws_bytes,
                               int batch, void* stream) {
  if (!x || !y || !ws) return fail(DS_ERR_INVALID_ARG, "NULL x, y or workspace");
  Plan P;
  ds_status r = plan_program(L, n, batch, P);
  if (r != DS_OK) return r;
  if (ws_bytes < P.total)
    return fail(DS_ERR_BUFFER_TOO_SMALL, "workspace has %zu bytes, needs %zu", ws_bytes, P.total);
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return fail(DS_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  if ((reinterpret_cast<uintptr_t>(x) & 15) != 0 || (reinterpret_cast<uintptr_t>(y) & 15) != 0)
    return fail(DS_ERR_ALIGNMENT, "x and y must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  unsigned char* base = static_cast<unsigned char*>(ws);
  uint32_t* amax = reinterpret_cast<uint32_t*>(base);
  std::vector<int32_t*> slot_ptr(P.n_slots, nullptr);
  std::vector<const uint32_t*> slot_amax(P.n_slots, nullptr);
  slot_ptr[0] = const_cast<int32_t*>(x);
  slot_ptr[1] = y;
  for (int s = 2; s < P.n_slots; ++s) slot_ptr[s] = reinterpret_cast<int32_t*>(base + P.slot_off[s]);

  // one reset per forward: the max|x| words and the split-reduction scratch (its
  // zero prefix is kept zero by the finalize kernels, larger regions are zeroed
  // before their layer)
  const size_t split_regions = P.any_side ? 2 : 1;
  r = cuda_check(cudaMemsetAsync(amax, 0, P.amax_bytes + split_regions * P.split_bytes, st), "workspace reset");
  if (r != DS_OK) return r;
  const Shape in0{L[0].C, L[0].H, L[0].W};
  r = cuda_check(launch_absmax(x, in0.elems() * batch, amax + n, st), "input max|x| pre-pass");
  if (r != DS_OK) return r;
  slot_amax[0] = amax + n;

  // two-stream schedule (one stream when the program has no independent neighbours, or when the
  // side stream's objects cannot be created)
  SideStream* S = nullptr;
  const bool two = P.any_side && side_resources((size_t)n + 1, S);
  auto on_side = [&](int i) { return two && i >= 0 && P.side[i]; };
  auto stream_of = [&](int i) { return on_side(i) ? S->s : st; };
  auto event_of = [&](int i) { return S->ev[i >= 0 ? i : n]; };
  if (two && P.signals[n]) {
    r = cuda_check(cudaEventRecord(event_of(-1), st), "workspace reset event");
    if (r != DS_OK) return r;
  }

  static const char* const kOpName[] = {"layer", "conv", "fc", "maxpool", "avgpool"};
  for (int i = 0; i < n; ++i) {
    const ds_layer& l = L[i];
    const int32_t* xin = slot_ptr[l.in];
    int32_t* yout = slot_ptr[l.out];
    NvtxRange nvtx_layer(kOpName[(l.op >= DS_OP_CONV && l.op <= DS_OP_AVGPOOL) ? l.op : 0], i);
    const cudaStream_t ls = stream_of(i);
    if (two)
      for (int j : P.deps[i])
        if (on_side(j) != on_side(i)) {
          r = cuda_check(cudaStreamWaitEvent(ls, event_of(j), 0), "layer dependency");
          if (r != DS_OK) return r;
        }
    unsigned char* split = base + P.amax_bytes + (on_side(i) ? P.split_bytes : 0);
    switch (l.op) {
      case DS_OP_CONV:
        r = conv_launch(xin, l.w, l.bias, l.aux >= 0 ? slot_ptr[l.aux] : nullptr, yout, batch, l.C, l.H, l.W,
                        l.K, l.R, l.S, l.stride, l.pad, l.flags, slot_amax[l.in], amax + i, ls,
                        P.split_bytes ? reinterpret_cast<int64_t*>(split) : nullptr, P.split_bytes);
        slot_amax[l.out] = amax + i;
        break;
      case DS_OP_FC:
        r = fc_launch(xin, l.w, l.bias, yout, batch, (int64_t)l.C * l.H * l.W, l.K, l.flags & DS_RELU,
                      slot_amax[l.in], amax + i, ls);
        slot_amax[l.out] = amax + i;
        break;
      case DS_OP_MAXPOOL:
        r = cuda_check(launch_maxpool(xin, yout, (int64_t)batch * l.C, l.H, l.W, P.out_shape[i].H,
                                      P.out_shape[i].W, l.R, l.S, l.stride, l.pad, ls),
                       "maxpool launch");
        slot_amax[l.out] = slot_amax[l.in];
        break;
      default:
        r = cuda_check(launch_avgpool_floor(xin, yout, (int64_t)batch * l.C, l.H, l.W, P.out_shape[i].H,
                                            P.out_shape[i].W, l.R, l.S, l.stride, ls),
                       "avgpool launch");
        slot_amax[l.out] = slot_amax[l.in];
        break;
    }
    if (r != DS_OK) return r;
    if (two && P.signals[i]) {
      r = cuda_check(cudaEventRecord(event_of(i), ls), "layer event");
      if (r != DS_OK) return r;
    }
  }
  if (two)
    for (int i = n - 1; i >= 0; --i)
      if (P.side[i]) {  // the caller's stream resumes after the side stream's last layer
        r = cuda_check(cudaStreamWaitEvent(st, event_of(i), 0), "side stream join");
        if (r != DS_OK) return r;
        break;
      }
  return DS_OK;
}

ds_status ds_shift_forward(const ds_layer* L, int n, const int32_t* x, int32_t* y, void* ws, size_t ws_bytes,
                           int batch, void* stream) {
  NvtxRange nvtx_range("ds_shift_forward");
  clear_error();
  try {
    return shift_forward(L, n, x, y, ws, ws_bytes, batch, stream);
  } catch (const std::exception&) {
    return fail(DS_ERR_UNSUPPORTED, "host memory allocation failed");
  }
}

}  // extern "C"
