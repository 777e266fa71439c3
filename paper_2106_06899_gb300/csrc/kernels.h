// kernels.h -- internal interface between the C-ABI layer (api.cu) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace topk {

// topk above this uses 32-row CTAs on the SIMT path (heap memory is
// topk x rows x 8 bytes of shared memory).
constexpr int kSimtSmallRowsMaxK = 128;
constexpr int kSimtMaxK = 512;
// tcgen05 attention path limit: 128 rows' heaps up to k = 137, units of 64 or
// 32 query rows up to 256 or 512 (heaps in shared memory)
constexpr int kTcMaxK = 512;

struct AttnArgs {
  const void* q;
  const void* k;
  const void* v;
  void* out;
  int B, H, Lq, Lk, d, topk, chunk, causal, dtype;
  int32_t* idx;
  float* score;
  // device scratch of the tcgen05 split kernel (attn_tc_workspace_bytes)
  void* workspace = nullptr;
  size_t workspace_bytes = 0;
  // Eq. 2's masks besides causal: the key count of each batch ([B] int32,
  // key j valid iff j < kv_len[b]) and a bit mask (bit j % 32 of word
  // b * mask_bs + h * mask_hs + i * ceil(Lk / 32) + j / 32, 1 = valid)
  const int32_t* kv_len = nullptr;
  const uint32_t* mask = nullptr;
  long long mask_bs = 0, mask_hs = 0;
};

struct FfnArgs {
  const void* x;
  const void* W1;
  const void* W2;
  float* out;
  int N, d_model, d_ff, topk;
  int32_t* idx;
  float* score;
  void* workspace;
  size_t workspace_bytes;
  // if set, the W2 gather (the last kernel) waits for this event first: the
  // host-buffer entry copies W2 while the earlier kernels run
  cudaEvent_t w2_ready = nullptr;
};

// Each launcher returns the number of kernel launches (> 0) on success,
// 0 if it does not serve the given shape, -1 on a CUDA error.
int attn_simt(const AttnArgs& a, cudaStream_t st);
int attn_tc(const AttnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st);
bool attn_tc_supports(const AttnArgs& a);
// Bytes of device scratch attn_tc needs for these arguments on a device with
// num_sms SMs: the split kernel parks each unit's kept keys for its
// epilogue warps (a fixed amount per CTA, nothing per query row); 0 otherwise.
size_t attn_tc_workspace_bytes(const AttnArgs& a, int num_sms);

size_t ffn_workspace_bytes(int N, int d_model, int d_ff, int topk);
int ffn_tc(const FfnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st);

// Backward pass for a cached kept set (bwd.cu).  idx/score are the forward
// pass's [rows][topk] cache (-1 / -inf = empty slot); dq [rows][d], dk and dv
// [B*H*Lk][d] are fp32; dout has the dtype of q (attention) or is fp32 (FF).
struct AttnBwdArgs {
  const void* q;
  const void* k;
  const void* v;
  const void* dout;
  const int32_t* idx;
  const float* score;
  float* dq;
  float* dk;
  float* dv;
  int B, H, Lq, Lk, d, topk, dtype;
  void* workspace;  // attn_bwd_workspace_bytes
};

struct FfnBwdArgs {
  const void* x;
  const void* W1;
  const void* W2;
  const float* dout;
  const int32_t* idx;
  const float* score;
  float* dx;
  float* dW1;
  float* dW2;
  int N, d_model, d_ff, topk;
  void* workspace;  // ffn_bwd_workspace_bytes
};

size_t attn_bwd_workspace_bytes(int B, int H, int Lq, int Lk, int topk);
size_t ffn_bwd_workspace_bytes(int N, int d_model, int d_ff, int topk);
bool attn_bwd_supports(int d, int dtype);
int attn_bwd(const AttnBwdArgs& a, int num_sms, cudaStream_t st);
int ffn_bwd(const FfnBwdArgs& a, int num_sms, cudaStream_t st);

// Plain attention (attn_plain.cu): Eq. 1 under the causal mask and key counts,
// bf16, d in {64, 128}; the workspace holds V^T (plain_workspace_bytes).
struct PlainArgs {
  const void* q;
  const void* k;
  const void* v;
  void* out;
  int B, H, Lq, Lk, d, causal;
  const int32_t* kv_len;
  void* workspace;
};
size_t plain_workspace_bytes(int B, int H, int Lk, int d);
int attn_plain(const PlainArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st);

// Dense FF (ffn_plain.cu): ReLU(x W1^T) W2 in d_ff slices of `chunk` keys, the
// two products in cuBLAS; the workspace holds one slice of H (bf16).
struct FfnPlainArgs {
  const void* x;
  const void* W1;
  const void* W2;
  float* out;
  int N, d_model, d_ff, chunk;
  void* workspace;
};
size_t ffn_plain_workspace_bytes(int N, int d_ff, int chunk);
int ffn_plain(const FfnPlainArgs& a, int num_sms, cudaStream_t st);

// Driver entry point for cuTensorMapEncodeTiled (resolved once, no libcuda link).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled_fn();

// 3-D bf16 tensor map [dim2][dim1][dim0] (dim0 innermost, contiguous) with a
// box of {64, box1, 1} and 128-byte swizzle.  Returns false on failure.
bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint64_t dim2,
                       uint32_t box1);

}  // namespace topk
