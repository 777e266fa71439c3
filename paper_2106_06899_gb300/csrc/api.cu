// api.cu -- the C ABI of libtopk.so (declared in include/topk_attention.h).
//
// Validates every argument before anything is enqueued, picks a kernel for
// the shape, and launches it on the caller's stream.  Device pointers are
// the caller's; the only state kept here is per-device: the device error
// word (OR-ed by kernels whose bounded waits ran out) and the SM count.
#include <atomic>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "topk_attention.h"
#include "kernels.h"

namespace topk {

namespace {

__device__ unsigned g_device_error;  // one word per device, OR of kDevErr* flags

constexpr int kMaxDevices = 64;
constexpr int kAssumedSms = 152;  // SMs of a GB300, for size queries made without a device
struct DeviceState {
  std::once_flag once;
  unsigned* error_word = nullptr;
  int num_sms = 0;
  int cc_major = 0, cc_minor = 0;
  bool ok = false;
};
DeviceState g_dev[kMaxDevices];

std::atomic<long long> g_wait_limit_us{0};
std::atomic<int> g_debug_skip_arrive{0};
thread_local int t_last_launches = 0;

DeviceState* device_state() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  DeviceState& s = g_dev[dev];
  std::call_once(s.once, [&s, dev]() {
    cudaDeviceProp p;
    if (cudaGetDeviceProperties(&p, dev) != cudaSuccess) return;
    s.num_sms = p.multiProcessorCount;
    s.cc_major = p.major;
    s.cc_minor = p.minor;
    void* addr = nullptr;
    if (cudaGetSymbolAddress(&addr, g_device_error) != cudaSuccess) return;
    s.error_word = static_cast<unsigned*>(addr);
    s.ok = true;
  });
  return s.ok ? &s : nullptr;
}

DevCtl make_ctl(DeviceState* s) {
  DevCtl c;
  c.error = s->error_word;
  const long long us = g_wait_limit_us.load();
  c.wait_limit_ns = static_cast<unsigned long long>(us > 0 ? us : 2000000LL) * 1000ull;
  c.debug_skip_arrive = g_debug_skip_arrive.load();
  return c;
}

// Device memory the library allocates itself (scratch, the staging buffers
// of the host-buffer calls) comes from one stream-ordered pool per device
// that keeps freed memory reserved for the next call, so a steady stream of
// calls of one shape maps device memory once instead of on every call.  Two
// non-blocking streams per device carry the host-buffer calls' copies, so
// that they overlap the kernels, and two more take the attention call's head
// slices in turn, so that the next slice's CTAs take the SMs that the
// previous slice's last, partial wave leaves idle.
struct HostPipe {
  std::once_flag once;
  cudaMemPool_t pool = nullptr;
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaStream_t comp[2] = {nullptr, nullptr};  // head slices alternate between these
  bool ok = false;
};
HostPipe g_pipe[kMaxDevices];

HostPipe* host_pipe() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  HostPipe& s = g_pipe[dev];
  std::call_once(s.once, [&s, dev]() {
    cudaMemPoolProps props;
    std::memset(&props, 0, sizeof props);
    props.allocType = cudaMemAllocationTypePinned;
    props.handleTypes = cudaMemHandleTypeNone;
    props.location.type = cudaMemLocationTypeDevice;
    props.location.id = dev;
    if (cudaMemPoolCreate(&s.pool, &props) != cudaSuccess) return;
    cuuint64_t keep = ~0ull;  // never hand freed memory back between calls
    if (cudaMemPoolSetAttribute(s.pool, cudaMemPoolAttrReleaseThreshold, &keep) != cudaSuccess) return;
    if (cudaStreamCreateWithFlags(&s.h2d, cudaStreamNonBlocking) != cudaSuccess) return;
    if (cudaStreamCreateWithFlags(&s.d2h, cudaStreamNonBlocking) != cudaSuccess) return;
    for (cudaStream_t& c : s.comp)
      if (cudaStreamCreateWithFlags(&c, cudaStreamNonBlocking) != cudaSuccess) return;
    s.ok = true;
  });
  return s.ok ? &s : nullptr;
}

bool pool_alloc(void** p, size_t bytes, cudaStream_t st) {
  HostPipe* hp = host_pipe();
  return hp && cudaMallocFromPoolAsync(p, bytes, hp->pool, st) == cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int validate_attn(const AttnArgs& a) {
  if (!a.q || !a.k || !a.v || !a.out) return TOPK_ERR_INVALID_ARG;
  if (a.B <= 0 || a.H <= 0 || a.Lq <= 0 || a.Lk <= 0 || a.d <= 0) return TOPK_ERR_INVALID_ARG;
  if (a.topk < 1 || a.topk > a.Lk || a.chunk < 1) return TOPK_ERR_INVALID_ARG;
  if (a.causal != 0 && a.causal != 1) return TOPK_ERR_INVALID_ARG;
  if (a.causal && a.Lq > a.Lk) return TOPK_ERR_INVALID_ARG;
  if (a.mask_bs < 0 || a.mask_hs < 0) return TOPK_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(a.mask) & 3u) return TOPK_ERR_UNSUPPORTED;
  if (a.kv_len && (reinterpret_cast<uintptr_t>(a.kv_len) & 3u)) return TOPK_ERR_UNSUPPORTED;
  if (a.dtype != TOPK_F32 && a.dtype != TOPK_BF16) return TOPK_ERR_INVALID_ARG;
  const long long BH = static_cast<long long>(a.B) * a.H;
  if (BH > (1 << 30) || static_cast<long long>(a.Lq) * BH > (1ll << 40)) return TOPK_ERR_UNSUPPORTED;
  if (a.topk > kSimtMaxK) return TOPK_ERR_UNSUPPORTED;
  if (a.dtype == TOPK_BF16 && a.d != 64 && a.d != 128) return TOPK_ERR_UNSUPPORTED;
  if (a.dtype == TOPK_F32 && a.d != 16 && a.d != 32 && a.d != 64 && a.d != 128) return TOPK_ERR_UNSUPPORTED;
  if (!aligned16(a.q) || !aligned16(a.k) || !aligned16(a.v) || !aligned16(a.out)) return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}

int run_attn(const AttnArgs& a, cudaStream_t st) {
  int rc = validate_attn(a);
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  const DevCtl ctl = make_ctl(dev);
  // k at least Lk keeps every valid key (Eq. 4 reduces to Eq. 1): without a
  // bit mask and without the selection as output, the plain kernel computes it
  // with no selection at all
  if (a.topk >= a.Lk && a.dtype == TOPK_BF16 && !a.mask && !a.idx && !a.score &&
      static_cast<long long>(a.B) * a.H <= 65535) {
    PlainArgs p{a.q, a.k, a.v, a.out, a.B, a.H, a.Lq, a.Lk, a.d, a.causal, a.kv_len, nullptr};
    void* pbuf = nullptr;
    if (!pool_alloc(&pbuf, plain_workspace_bytes(a.B, a.H, a.Lk, a.d), st)) return TOPK_ERR_CUDA;
    p.workspace = pbuf;
    const int n = attn_plain(p, ctl, dev->num_sms, st);
    cudaFreeAsync(pbuf, st);
    if (n < 0) return TOPK_ERR_CUDA;
    if (n > 0) {
      t_last_launches = n;
      return TOPK_OK;
    }
  }
  const size_t ws = attn_tc_workspace_bytes(a, dev->num_sms);
  void* buf = nullptr;
  if (ws && !pool_alloc(&buf, ws, st)) return TOPK_ERR_CUDA;
  AttnArgs b = a;
  b.workspace = buf;
  b.workspace_bytes = ws;
  int n = attn_tc(b, ctl, dev->num_sms, st);
  if (buf) cudaFreeAsync(buf, st);
  if (n == 0) n = attn_simt(a, st);
  if (n == 0) return TOPK_ERR_UNSUPPORTED;
  if (n < 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

int validate_ffn(const FfnArgs& a) {
  if (!a.x || !a.W1 || !a.W2 || !a.out) return TOPK_ERR_INVALID_ARG;
  if (a.N <= 0 || a.d_model <= 0 || a.d_ff <= 0) return TOPK_ERR_INVALID_ARG;
  if (a.topk < 1 || a.topk > a.d_ff) return TOPK_ERR_INVALID_ARG;
  if (a.d_model % 64 != 0 || a.d_model > 4096) return TOPK_ERR_UNSUPPORTED;
  if (a.topk > 1024) return TOPK_ERR_UNSUPPORTED;
  if (!aligned16(a.x) || !aligned16(a.W1) || !aligned16(a.W2) || !aligned16(a.out)) return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}

int run_ffn(FfnArgs a, cudaStream_t st) {
  int rc = validate_ffn(a);
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  const DevCtl ctl = make_ctl(dev);
  const size_t ws = ffn_workspace_bytes(a.N, a.d_model, a.d_ff, a.topk);
  void* buf = nullptr;
  if (ws && !pool_alloc(&buf, ws, st)) return TOPK_ERR_CUDA;
  a.workspace = buf;
  a.workspace_bytes = ws;
  int n = ffn_tc(a, ctl, dev->num_sms, st);
  if (buf) cudaFreeAsync(buf, st);
  if (n == 0) return TOPK_ERR_UNSUPPORTED;
  if (n < 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

size_t elem_bytes(int dtype) { return dtype == TOPK_F32 ? 4 : 2; }

int validate_plain(const PlainArgs& a, int chunk, int dtype) {
  if (!a.q || !a.k || !a.v || !a.out) return TOPK_ERR_INVALID_ARG;
  if (a.B <= 0 || a.H <= 0 || a.Lq <= 0 || a.Lk <= 0 || a.d <= 0 || chunk < 1) return TOPK_ERR_INVALID_ARG;
  if (a.causal != 0 && a.causal != 1) return TOPK_ERR_INVALID_ARG;
  if (a.causal && a.Lq > a.Lk) return TOPK_ERR_INVALID_ARG;
  if (dtype != TOPK_F32 && dtype != TOPK_BF16) return TOPK_ERR_INVALID_ARG;
  if (dtype != TOPK_BF16 || (a.d != 64 && a.d != 128)) return TOPK_ERR_UNSUPPORTED;
  if (static_cast<long long>(a.B) * a.H > 65535) return TOPK_ERR_UNSUPPORTED;
  if (!aligned16(a.q) || !aligned16(a.k) || !aligned16(a.v) || !aligned16(a.out)) return TOPK_ERR_UNSUPPORTED;
  if (a.kv_len && (reinterpret_cast<uintptr_t>(a.kv_len) & 3u)) return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}

// Backward pass (bwd.cu): the cache width, the entry and bucket counts are
// bounded so that slots and offsets fit in 32-bit integers.
constexpr int kBwdMaxK = 2048;

int validate_attn_bwd(const AttnBwdArgs& a) {
  if (!a.q || !a.k || !a.v || !a.dout || !a.idx || !a.score || !a.dq || !a.dk || !a.dv) return TOPK_ERR_INVALID_ARG;
  if (a.B <= 0 || a.H <= 0 || a.Lq <= 0 || a.Lk <= 0 || a.d <= 0) return TOPK_ERR_INVALID_ARG;
  if (a.topk < 1 || a.topk > a.Lk) return TOPK_ERR_INVALID_ARG;
  if (a.dtype != TOPK_F32 && a.dtype != TOPK_BF16) return TOPK_ERR_INVALID_ARG;
  if (a.topk > kBwdMaxK || !attn_bwd_supports(a.d, a.dtype)) return TOPK_ERR_UNSUPPORTED;
  const long long BH = static_cast<long long>(a.B) * a.H;
  if (BH * a.Lq * a.topk >= (1ll << 31) || BH * a.Lk >= (1ll << 31)) return TOPK_ERR_UNSUPPORTED;
  for (const void* p : {a.q, a.k, a.v, a.dout, static_cast<const void*>(a.dq), static_cast<const void*>(a.dk),
                        static_cast<const void*>(a.dv)})
    if (!aligned16(p)) return TOPK_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(a.idx) & 3u) || (reinterpret_cast<uintptr_t>(a.score) & 3u))
    return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}

int validate_ffn_bwd(const FfnBwdArgs& a) {
  if (!a.x || !a.W1 || !a.W2 || !a.dout || !a.idx || !a.score || !a.dx || !a.dW1 || !a.dW2)
    return TOPK_ERR_INVALID_ARG;
  if (a.N <= 0 || a.d_model <= 0 || a.d_ff <= 0) return TOPK_ERR_INVALID_ARG;
  if (a.topk < 1 || a.topk > a.d_ff) return TOPK_ERR_INVALID_ARG;
  if (a.d_model % 64 != 0 || a.d_model > 2048) return TOPK_ERR_UNSUPPORTED;
  if (static_cast<long long>(a.N) * a.topk >= (1ll << 31)) return TOPK_ERR_UNSUPPORTED;
  for (const void* p : {a.x, a.W1, a.W2, static_cast<const void*>(a.dout), static_cast<const void*>(a.dx),
                        static_cast<const void*>(a.dW1), static_cast<const void*>(a.dW2)})
    if (!aligned16(p)) return TOPK_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(a.idx) & 3u) || (reinterpret_cast<uintptr_t>(a.score) & 3u))
    return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}

template <typename Args, typename Size, typename Run>
int run_bwd(Args a, int rc, Size size, Run launch, cudaStream_t st) {
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  void* buf = nullptr;
  if (!pool_alloc(&buf, size(a), st)) return TOPK_ERR_CUDA;
  a.workspace = buf;
  const int n = launch(a, dev->num_sms, st);
  cudaFreeAsync(buf, st);
  if (n == 0) return TOPK_ERR_UNSUPPORTED;
  if (n < 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

}  // namespace

EncodeTiledFn encode_tiled_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, []() {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint64_t dim2,
                       uint32_t box1) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {dim0, dim1, dim2};
  cuuint64_t strides[2] = {dim0 * 2, dim0 * dim1 * 2};
  cuuint32_t box[3] = {64, box1, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace topk

using namespace topk;

extern "C" {

int topk_attn_fwd(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk, int d,
                  int topk, int chunk, int causal, int dtype, void* stream) {
  AttnArgs a{q, k, v, out, B, H, Lq, Lk, d, topk, chunk, causal, dtype, nullptr, nullptr};
  return run_attn(a, static_cast<cudaStream_t>(stream));
}

int topk_attn_fwd_indices(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                          int d, int topk, int chunk, int causal, int dtype, int32_t* idx, float* score,
                          void* stream) {
  if ((idx && !aligned16(idx)) || (score && !aligned16(score))) return TOPK_ERR_UNSUPPORTED;
  AttnArgs a{q, k, v, out, B, H, Lq, Lk, d, topk, chunk, causal, dtype, idx, score};
  return run_attn(a, static_cast<cudaStream_t>(stream));
}

int topk_attn_fwd_masked(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                         int d, int topk, int chunk, int causal, const int32_t* kv_len, const uint32_t* mask,
                         long long mask_batch_stride, long long mask_head_stride, int dtype, int32_t* idx,
                         float* score, void* stream) {
  if ((idx && !aligned16(idx)) || (score && !aligned16(score))) return TOPK_ERR_UNSUPPORTED;
  AttnArgs a{q, k, v, out, B, H, Lq, Lk, d, topk, chunk, causal, dtype, idx, score};
  a.kv_len = kv_len;
  a.mask = mask;
  a.mask_bs = mask_batch_stride;
  a.mask_hs = mask_head_stride;
  return run_attn(a, static_cast<cudaStream_t>(stream));
}

int topk_ffn_fwd(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff, int topk,
                 void* stream) {
  FfnArgs a{x, W1, W2, static_cast<float*>(out), N, d_model, d_ff, topk, nullptr, nullptr, nullptr, 0};
  return run_ffn(a, static_cast<cudaStream_t>(stream));
}

int topk_ffn_fwd_indices(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                         int topk, int32_t* idx, float* score, void* stream) {
  FfnArgs a{x, W1, W2, static_cast<float*>(out), N, d_model, d_ff, topk, idx, score, nullptr, 0};
  return run_ffn(a, static_cast<cudaStream_t>(stream));
}

int topk_vanilla_attn_fwd(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                          int d, int chunk, int causal, const int32_t* kv_len, int dtype, void* stream) {
  PlainArgs a{q, k, v, out, B, H, Lq, Lk, d, causal, kv_len, nullptr};
  int rc = validate_plain(a, chunk, dtype);
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* buf = nullptr;
  if (!pool_alloc(&buf, plain_workspace_bytes(B, H, Lk, d), st)) return TOPK_ERR_CUDA;
  a.workspace = buf;
  const int n = attn_plain(a, make_ctl(dev), dev->num_sms, st);
  cudaFreeAsync(buf, st);
  if (n == 0) return TOPK_ERR_UNSUPPORTED;
  if (n < 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

size_t topk_vanilla_attn_workspace_bytes(int B, int H, int Lq, int Lk, int d, int dtype) {
  PlainArgs a{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
              reinterpret_cast<void*>(16), B, H, Lq, Lk, d, 0, nullptr, nullptr};
  if (validate_plain(a, 1, dtype) != TOPK_OK) return 0;
  return plain_workspace_bytes(B, H, Lk, d);
}

namespace {
int validate_ffn_plain(const FfnPlainArgs& a) {
  if (!a.x || !a.W1 || !a.W2 || !a.out) return TOPK_ERR_INVALID_ARG;
  if (a.N <= 0 || a.d_model <= 0 || a.d_ff <= 0 || a.chunk < 1) return TOPK_ERR_INVALID_ARG;
  if (a.d_model % 8 != 0) return TOPK_ERR_UNSUPPORTED;
  const long long c = a.chunk < a.d_ff ? a.chunk : a.d_ff;
  if (c % 8 != 0 && c != a.d_ff) return TOPK_ERR_UNSUPPORTED;  // H rows stay 16-byte aligned
  if ((static_cast<long long>(a.N) * c) % 8 != 0) return TOPK_ERR_UNSUPPORTED;
  if (!aligned16(a.x) || !aligned16(a.W1) || !aligned16(a.W2) || !aligned16(a.out)) return TOPK_ERR_UNSUPPORTED;
  return TOPK_OK;
}
}  // namespace

int topk_vanilla_ffn_fwd(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                         int chunk, void* stream) {
  FfnPlainArgs a{x, W1, W2, static_cast<float*>(out), N, d_model, d_ff, chunk, nullptr};
  int rc = validate_ffn_plain(a);
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* buf = nullptr;
  if (!pool_alloc(&buf, ffn_plain_workspace_bytes(N, d_ff, chunk), st)) return TOPK_ERR_CUDA;
  a.workspace = buf;
  const int n = ffn_plain(a, dev->num_sms, st);
  cudaFreeAsync(buf, st);
  if (n <= 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

size_t topk_vanilla_ffn_workspace_bytes(int N, int d_model, int d_ff, int chunk) {
  FfnPlainArgs a{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
                 reinterpret_cast<float*>(16), N, d_model, d_ff, chunk, nullptr};
  if (validate_ffn_plain(a) != TOPK_OK) return 0;
  return ffn_plain_workspace_bytes(N, d_ff, chunk);
}

int topk_attn_bwd(const void* q, const void* k, const void* v, const void* dout, const int32_t* idx,
                  const float* score, float* dq, float* dk, float* dv, int B, int H, int Lq, int Lk, int d,
                  int topk, int dtype, void* stream) {
  AttnBwdArgs a{q, k, v, dout, idx, score, dq, dk, dv, B, H, Lq, Lk, d, topk, dtype, nullptr};
  return run_bwd(
      a, validate_attn_bwd(a),
      [](const AttnBwdArgs& x) { return attn_bwd_workspace_bytes(x.B, x.H, x.Lq, x.Lk, x.topk); },
      [](const AttnBwdArgs& x, int sms, cudaStream_t s) { return attn_bwd(x, sms, s); },
      static_cast<cudaStream_t>(stream));
}

int topk_ffn_bwd(const void* x, const void* W1, const void* W2, const float* dout, const int32_t* idx,
                 const float* score, float* dx, float* dW1, float* dW2, int N, int d_model, int d_ff, int topk,
                 void* stream) {
  FfnBwdArgs a{x, W1, W2, dout, idx, score, dx, dW1, dW2, N, d_model, d_ff, topk, nullptr};
  return run_bwd(
      a, validate_ffn_bwd(a), [](const FfnBwdArgs& y) { return ffn_bwd_workspace_bytes(y.N, y.d_model, y.d_ff, y.topk); },
      [](const FfnBwdArgs& y, int sms, cudaStream_t s) { return ffn_bwd(y, sms, s); },
      static_cast<cudaStream_t>(stream));
}

size_t topk_attn_bwd_workspace_bytes(int B, int H, int Lq, int Lk, int d, int topk, int dtype) {
  void* p = reinterpret_cast<void*>(16);
  float* f = reinterpret_cast<float*>(16);
  AttnBwdArgs a{p, p, p, p, reinterpret_cast<const int32_t*>(16), f, f, f, f, B, H, Lq, Lk, d, topk, dtype, nullptr};
  if (validate_attn_bwd(a) != TOPK_OK) return 0;
  return attn_bwd_workspace_bytes(B, H, Lq, Lk, topk);
}

size_t topk_ffn_bwd_workspace_bytes(int N, int d_model, int d_ff, int topk) {
  void* p = reinterpret_cast<void*>(16);
  float* f = reinterpret_cast<float*>(16);
  FfnBwdArgs a{p, p, p, f, reinterpret_cast<const int32_t*>(16), f, f, f, f, N, d_model, d_ff, topk, nullptr};
  if (validate_ffn_bwd(a) != TOPK_OK) return 0;
  return ffn_bwd_workspace_bytes(N, d_model, d_ff, topk);
}

size_t topk_attn_workspace_bytes(int B, int H, int Lq, int Lk, int d, int topk, int chunk, int dtype) {
  AttnArgs a{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
             reinterpret_cast<void*>(16), B, H, Lq, Lk, d, topk, chunk, 0, dtype, nullptr, nullptr};
  if (validate_attn(a) != TOPK_OK) return 0;
  // sized for the current device (the SM count the launch uses); for a
  // GB300 (152 SMs) when none is visible
  const DeviceState* dev = device_state();
  return attn_tc_workspace_bytes(a, dev ? dev->num_sms : kAssumedSms);
}

size_t topk_ffn_workspace_bytes(int N, int d_model, int d_ff, int topk) {
  FfnArgs a{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
            reinterpret_cast<float*>(16), N, d_model, d_ff, topk, nullptr, nullptr, nullptr, 0};
  if (validate_ffn(a) != TOPK_OK) return 0;
  return ffn_workspace_bytes(N, d_model, d_ff, topk);
}

namespace {
// After a synchronising host-buffer call: report any device-side error flag.
int host_call_status(int rc) {
  if (rc != TOPK_OK) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  unsigned word = 0;
  if (cudaMemcpy(&word, dev->error_word, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return TOPK_ERR_CUDA;
  if (!word) return TOPK_OK;
  const unsigned zero = 0;
  cudaMemcpy(dev->error_word, &zero, sizeof zero, cudaMemcpyHostToDevice);
  return (word & kDevErrTimeout) ? TOPK_ERR_TIMEOUT : TOPK_ERR_WORKSPACE;
}
}  // namespace

// Head slices of a host-buffer attention call: about 6 or more 128-query
// tiles per SM in each slice (the persistent launch of a slice then loses
// little to its last, partial wave), at most 8 slices.  More slices expose
// less copy time at the two ends (the first slice's inputs, the last
// slice's output).
constexpr int kHostSlicesMax = 8;

int topk_attn_fwd_host(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk, int d,
                       int topk, int chunk, int causal, int dtype, void* stream) {
  if (!q || !k || !v || !out) return TOPK_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || Lq <= 0 || Lk <= 0 || d <= 0) return TOPK_ERR_INVALID_ARG;
  AttnArgs chk{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
               reinterpret_cast<void*>(16), B, H, Lq, Lk, d, topk, chunk, causal, dtype, nullptr, nullptr};
  int rc = validate_attn(chk);
  if (rc) return rc;
  DeviceState* dev = device_state();
  HostPipe* hp = host_pipe();
  if (!dev || !hp) return TOPK_ERR_NO_DEVICE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t eb = elem_bytes(dtype);
  const int BH = B * H;
  const size_t qh = static_cast<size_t>(Lq) * d * eb, kh = static_cast<size_t>(Lk) * d * eb;
  const long long tiles = static_cast<long long>(BH) * ((Lq + 127) / 128);
  int P = static_cast<int>(tiles / (6LL * dev->num_sms));
  P = P < 1 ? 1 : (P > BH ? BH : (P > kHostSlicesMax ? kHostSlicesMax : P));

  void *dq = nullptr, *dk = nullptr, *dv = nullptr, *dout = nullptr;
  cudaEvent_t ready = nullptr, h2d_done = nullptr, d2h_done = nullptr, comp_done[2] = {nullptr, nullptr};
  cudaEvent_t ev_in[kHostSlicesMax] = {}, ev_out[kHostSlicesMax] = {};
  auto mk = [](cudaEvent_t* e) { return cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess; };
  bool good = pool_alloc(&dq, BH * qh, st) && pool_alloc(&dk, BH * kh, st) && pool_alloc(&dv, BH * kh, st) &&
              pool_alloc(&dout, BH * qh, st) && mk(&ready) && mk(&h2d_done) && mk(&d2h_done) &&
              mk(&comp_done[0]) && mk(&comp_done[1]);
  for (int s = 0; good && s < P; ++s) good = mk(&ev_in[s]) && mk(&ev_out[s]);
  // the library streams start once the allocations on `st` are in place
  good = good && cudaEventRecord(ready, st) == cudaSuccess;
  for (cudaStream_t w : {hp->h2d, hp->d2h, hp->comp[0], hp->comp[1]})
    good = good && cudaStreamWaitEvent(w, ready, 0) == cudaSuccess;
  if (!good) rc = TOPK_ERR_CUDA;
  // slice s: its inputs on the h2d stream, its launch on compute stream
  // s % 2 after them, its output on the d2h stream after the launch; the
  // copies of slices s + 1 and s - 1 overlap the kernel of slice s, and the
  // kernel of slice s + 1 starts on the SMs that slice s frees
  int launches = 0;
  for (int s = 0; rc == TOPK_OK && s < P; ++s) {
    const size_t h0 = static_cast<size_t>(static_cast<long long>(BH) * s / P);
    const size_t h1 = static_cast<size_t>(static_cast<long long>(BH) * (s + 1) / P);
    const size_t nh = h1 - h0;
    uint8_t* sq = static_cast<uint8_t*>(dq) + h0 * qh;
    uint8_t* sk = static_cast<uint8_t*>(dk) + h0 * kh;
    uint8_t* sv = static_cast<uint8_t*>(dv) + h0 * kh;
    uint8_t* so = static_cast<uint8_t*>(dout) + h0 * qh;
    if (cudaMemcpyAsync(sq, static_cast<const uint8_t*>(q) + h0 * qh, nh * qh, cudaMemcpyHostToDevice, hp->h2d) !=
            cudaSuccess ||
        cudaMemcpyAsync(sk, static_cast<const uint8_t*>(k) + h0 * kh, nh * kh, cudaMemcpyHostToDevice, hp->h2d) !=
            cudaSuccess ||
        cudaMemcpyAsync(sv, static_cast<const uint8_t*>(v) + h0 * kh, nh * kh, cudaMemcpyHostToDevice, hp->h2d) !=
            cudaSuccess ||
        cudaEventRecord(ev_in[s], hp->h2d) != cudaSuccess) {
      rc = TOPK_ERR_CUDA;
      break;
    }
    cudaStream_t cs = hp->comp[s & 1];
    if (cudaStreamWaitEvent(cs, ev_in[s], 0) != cudaSuccess) {
      rc = TOPK_ERR_CUDA;
      break;
    }
    rc = topk_attn_fwd(sq, sk, sv, so, 1, static_cast<int>(nh), Lq, Lk, d, topk, chunk, causal, dtype, cs);
    if (rc != TOPK_OK) break;
    launches += t_last_launches;
    if (cudaEventRecord(ev_out[s], cs) != cudaSuccess || cudaStreamWaitEvent(hp->d2h, ev_out[s], 0) != cudaSuccess ||
        cudaMemcpyAsync(static_cast<uint8_t*>(out) + h0 * qh, so, nh * qh, cudaMemcpyDeviceToHost, hp->d2h) !=
            cudaSuccess) {
      rc = TOPK_ERR_CUDA;
      break;
    }
  }
  // the buffers go back to the pool on `st` only after the copy and
  // compute streams are done with everything enqueued above
  bool joined = h2d_done && d2h_done && comp_done[0] && comp_done[1] &&
                cudaEventRecord(h2d_done, hp->h2d) == cudaSuccess &&
                cudaEventRecord(d2h_done, hp->d2h) == cudaSuccess &&
                cudaEventRecord(comp_done[0], hp->comp[0]) == cudaSuccess &&
                cudaEventRecord(comp_done[1], hp->comp[1]) == cudaSuccess;
  for (cudaEvent_t e : {h2d_done, d2h_done, comp_done[0], comp_done[1]})
    joined = joined && cudaStreamWaitEvent(st, e, 0) == cudaSuccess;
  if (!joined) {
    for (cudaStream_t w : {hp->h2d, hp->d2h, hp->comp[0], hp->comp[1]}) cudaStreamSynchronize(w);
    if (rc == TOPK_OK) rc = TOPK_ERR_CUDA;
  }
  if (dq) cudaFreeAsync(dq, st);
  if (dk) cudaFreeAsync(dk, st);
  if (dv) cudaFreeAsync(dv, st);
  if (dout) cudaFreeAsync(dout, st);
  if (cudaStreamSynchronize(st) != cudaSuccess && rc == TOPK_OK) rc = TOPK_ERR_CUDA;
  for (cudaEvent_t e : {ready, h2d_done, d2h_done, comp_done[0], comp_done[1]})
    if (e) cudaEventDestroy(e);
  for (int s = 0; s < P; ++s) {
    if (ev_in[s]) cudaEventDestroy(ev_in[s]);
    if (ev_out[s]) cudaEventDestroy(ev_out[s]);
  }
  t_last_launches = launches;
  return host_call_status(rc);
}

int topk_ffn_fwd_host(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                      int topk, void* stream) {
  if (!x || !W1 || !W2 || !out) return TOPK_ERR_INVALID_ARG;
  FfnArgs chk{reinterpret_cast<void*>(16), reinterpret_cast<void*>(16), reinterpret_cast<void*>(16),
              reinterpret_cast<float*>(16), N, d_model, d_ff, topk, nullptr, nullptr, nullptr, 0};
  int rc = validate_ffn(chk);
  if (rc) return rc;
  HostPipe* hp = host_pipe();
  if (!hp) return TOPK_ERR_NO_DEVICE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t xb = static_cast<size_t>(N) * d_model * 2, wb = static_cast<size_t>(d_ff) * d_model * 2;
  const size_t ob = static_cast<size_t>(N) * d_model * 4;
  void *dx = nullptr, *d1 = nullptr, *d2 = nullptr, *dout = nullptr;
  cudaEvent_t ready = nullptr, in_ready = nullptr, w2_ready = nullptr, h2d_done = nullptr;
  auto mk = [](cudaEvent_t* e) { return cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess; };
  bool good = pool_alloc(&dx, xb, st) && pool_alloc(&d1, wb, st) && pool_alloc(&d2, wb, st) &&
              pool_alloc(&dout, ob, st) && mk(&ready) && mk(&in_ready) && mk(&w2_ready) && mk(&h2d_done);
  // x and W1 first (the score kernel needs them), then W2, which only the
  // last kernel (the gather) reads: its copy overlaps the first two kernels
  good = good && cudaEventRecord(ready, st) == cudaSuccess && cudaStreamWaitEvent(hp->h2d, ready, 0) == cudaSuccess &&
         cudaMemcpyAsync(dx, x, xb, cudaMemcpyHostToDevice, hp->h2d) == cudaSuccess &&
         cudaMemcpyAsync(d1, W1, wb, cudaMemcpyHostToDevice, hp->h2d) == cudaSuccess &&
         cudaEventRecord(in_ready, hp->h2d) == cudaSuccess &&
         cudaMemcpyAsync(d2, W2, wb, cudaMemcpyHostToDevice, hp->h2d) == cudaSuccess &&
         cudaEventRecord(w2_ready, hp->h2d) == cudaSuccess && cudaStreamWaitEvent(st, in_ready, 0) == cudaSuccess;
  if (!good) {
    rc = TOPK_ERR_CUDA;
  } else {
    FfnArgs a{dx, d1, d2, static_cast<float*>(dout), N, d_model, d_ff, topk, nullptr, nullptr, nullptr, 0};
    a.w2_ready = w2_ready;
    rc = run_ffn(a, st);
    if (rc == TOPK_OK && cudaMemcpyAsync(out, dout, ob, cudaMemcpyDeviceToHost, st) != cudaSuccess)
      rc = TOPK_ERR_CUDA;
  }
  const int launches = t_last_launches;
  // every copy enqueued on the h2d stream ends before the buffers are freed
  if (!(h2d_done && cudaEventRecord(h2d_done, hp->h2d) == cudaSuccess &&
        cudaStreamWaitEvent(st, h2d_done, 0) == cudaSuccess)) {
    cudaStreamSynchronize(hp->h2d);
    if (rc == TOPK_OK) rc = TOPK_ERR_CUDA;
  }
  if (dx) cudaFreeAsync(dx, st);
  if (d1) cudaFreeAsync(d1, st);
  if (d2) cudaFreeAsync(d2, st);
  if (dout) cudaFreeAsync(dout, st);
  if (cudaStreamSynchronize(st) != cudaSuccess && rc == TOPK_OK) rc = TOPK_ERR_CUDA;
  for (cudaEvent_t e : {ready, in_ready, w2_ready, h2d_done})
    if (e) cudaEventDestroy(e);
  t_last_launches = launches;
  return host_call_status(rc);
}

}  // extern "C"

// ---------------------------------------------------------------- no-allocation FF entry
namespace topk {
namespace {

// Scratch of topk_ffn_fwd_noalloc: part of the module image, held by every
// device that loads the library until the process exits.
static __device__ __align__(256) unsigned char g_ffn_noalloc_scratch[TOPK_FFN_NOALLOC_SCRATCH_BYTES];

struct NoAllocState {
  std::once_flag once;
  void* ptr = nullptr;
};
NoAllocState g_noalloc[kMaxDevices];

// Device address of the scratch array on the current device (looked up once
// per device, with that device current).  Host code must not use the array's
// name as an address: on the host it is only a stand-in for the symbol.
void* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  NoAllocState& s = g_noalloc[dev];
  std::call_once(s.once, [&s]() {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_ffn_noalloc_scratch) == cudaSuccess) s.ptr = p;
  });
  return s.ptr;
}

}  // namespace
}  // namespace topk

extern "C" {

int topk_ffn_fwd_noalloc(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                         int topk, void* stream) {
  FfnArgs a{x, W1, W2, static_cast<float*>(out), N, d_model, d_ff, topk, nullptr, nullptr, nullptr, 0};
  int rc = validate_ffn(a);
  if (rc) return rc;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  if (dev->cc_major != 10 || dev->cc_minor != 3) return TOPK_ERR_NO_DEVICE;
  if (ffn_workspace_bytes(N, d_model, d_ff, topk) > TOPK_FFN_NOALLOC_SCRATCH_BYTES) return TOPK_ERR_SCRATCH_LIMIT;
  void* scratch = noalloc_scratch();
  if (!scratch) return TOPK_ERR_CUDA;
  a.workspace = scratch;
  a.workspace_bytes = TOPK_FFN_NOALLOC_SCRATCH_BYTES;
  const int n = ffn_tc(a, make_ctl(dev), dev->num_sms, static_cast<cudaStream_t>(stream));
  if (n == 0) return TOPK_ERR_UNSUPPORTED;
  if (n < 0) return TOPK_ERR_CUDA;
  t_last_launches = n;
  return TOPK_OK;
}

int topk_check(void* stream) {
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return TOPK_ERR_CUDA;
  DeviceState* dev = device_state();
  if (!dev) return TOPK_ERR_NO_DEVICE;
  unsigned word = 0;
  if (cudaMemcpy(&word, dev->error_word, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return TOPK_ERR_CUDA;
  if (word) {
    const unsigned zero = 0;
    if (cudaMemcpy(dev->error_word, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess)
      return TOPK_ERR_CUDA;
  }
  if (word & kDevErrTimeout) return TOPK_ERR_TIMEOUT;
  if (word & kDevErrWorkspace) return TOPK_ERR_WORKSPACE;
  return TOPK_OK;
}

const char* topk_error_string(int code) {
  switch (code) {
    case TOPK_OK: return "success";
    case TOPK_ERR_INVALID_ARG: return "invalid argument";
    case TOPK_ERR_UNSUPPORTED: return "unsupported shape, dtype, topk or alignment";
    case TOPK_ERR_CUDA: return "CUDA error";
    case TOPK_ERR_TIMEOUT: return "device pipeline wait timed out; outputs invalid";
    case TOPK_ERR_WORKSPACE: return "per-row candidate list overflowed; outputs invalid";
    case TOPK_ERR_NO_DEVICE: return "no usable sm_103 device";
    case TOPK_ERR_SCRATCH_LIMIT: return "problem needs more scratch than the fixed no-allocation buffer holds";
    default: return "unknown error code";
  }
}

int topk_last_launch_count(void) { return t_last_launches; }

long long topk_set_wait_limit_us(long long us) { return g_wait_limit_us.exchange(us < 0 ? 0 : us); }

// Testing hook: makes the tcgen05 attention producer withhold its second key
// tile so that the consumers' bounded waits run out; returns the previous
// setting.
int topk_debug_skip_arrive(int on) { return g_debug_skip_arrive.exchange(on ? 1 : 0); }

int topk_pool_usage(size_t* used_high, size_t* reserved, int reset_high) {
  HostPipe* hp = host_pipe();
  if (!hp) return TOPK_ERR_NO_DEVICE;
  cuuint64_t hi = 0, res = 0;
  if (cudaMemPoolGetAttribute(hp->pool, cudaMemPoolAttrUsedMemHigh, &hi) != cudaSuccess ||
      cudaMemPoolGetAttribute(hp->pool, cudaMemPoolAttrReservedMemCurrent, &res) != cudaSuccess)
    return TOPK_ERR_CUDA;
  if (used_high) *used_high = static_cast<size_t>(hi);
  if (reserved) *reserved = static_cast<size_t>(res);
  if (reset_high) {
    cuuint64_t zero = 0;  // the only value the high-water attributes accept
    if (cudaMemPoolSetAttribute(hp->pool, cudaMemPoolAttrUsedMemHigh, &zero) != cudaSuccess) return TOPK_ERR_CUDA;
  }
  return TOPK_OK;
}

int topk_pool_trim(void) {
  HostPipe* hp = host_pipe();
  if (!hp) return TOPK_ERR_NO_DEVICE;
  return cudaMemPoolTrimTo(hp->pool, 0) == cudaSuccess ? TOPK_OK : TOPK_ERR_CUDA;
}

}  // extern "C"
