// ffn_plain.cu -- the dense feed-forward layer (Eq. 3 without top-k:
// out = ReLU(x W1^T) W2), the comparison path for the top-k FF layer (Sec. 3).
//
// Both products are plain GEMMs and run in cuBLAS (bf16 inputs, fp32
// accumulation).  d_ff is taken in slices of `chunk` keys, as the paper chunks
// to bound memory: per slice the hidden activations H = x W1_s^T [N, chunk]
// are written as bf16, ReLU is applied in place (the kernel below), and
// out += H W2_s accumulates in fp32.
#include <cublas_v2.h>
#include <cuda_bf16.h>

#include <mutex>

#include "kernels.h"

namespace topk {

namespace {

__global__ void relu_bf16_kernel(__nv_bfloat16* __restrict__ h, long long n8) {
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n8; i += stride) {
    uint4 u = reinterpret_cast<uint4*>(h)[i];
    uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      // bf16 sign bits 15 and 31: a negative half becomes +0
      if (w[e] & 0x8000u) w[e] &= 0xffff0000u;
      if (w[e] & 0x80000000u) w[e] &= 0x0000ffffu;
    }
    reinterpret_cast<uint4*>(h)[i] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

constexpr int kMaxDev = 64;
struct Blas {
  std::once_flag once;
  std::mutex mu;  // a cuBLAS handle serves one call at a time
  cublasHandle_t h = nullptr;
  bool ok = false;
};
Blas g_blas[kMaxDev];

Blas* blas() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return nullptr;
  Blas& b = g_blas[dev];
  std::call_once(b.once, [&b]() { b.ok = cublasCreate(&b.h) == CUBLAS_STATUS_SUCCESS; });
  return b.ok ? &b : nullptr;
}

}  // namespace

size_t ffn_plain_workspace_bytes(int N, int d_ff, int chunk) {
  const long long c = chunk < d_ff ? chunk : d_ff;
  return static_cast<size_t>(N) * c * 2;
}

int ffn_plain(const FfnPlainArgs& a, int num_sms, cudaStream_t st) {
  Blas* b = blas();
  if (!b) return -1;
  std::lock_guard<std::mutex> lock(b->mu);
  if (cublasSetStream(b->h, st) != CUBLAS_STATUS_SUCCESS) return -1;
  const int C = a.chunk < a.d_ff ? a.chunk : a.d_ff;
  const float one = 1.f, zero = 0.f;
  __nv_bfloat16* H = static_cast<__nv_bfloat16*>(a.workspace);
  const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(a.x);
  const __nv_bfloat16* W1 = static_cast<const __nv_bfloat16*>(a.W1);
  const __nv_bfloat16* W2 = static_cast<const __nv_bfloat16*>(a.W2);
  int launches = 0;
  for (int s0 = 0; s0 < a.d_ff; s0 += C) {
    const int c = a.d_ff - s0 < C ? a.d_ff - s0 : C;
    // column-major view: H^T [c, N] = W1_s [c, dm] (stored as dm x c) ^T * x^T [dm, N]
    if (cublasGemmEx(b->h, CUBLAS_OP_T, CUBLAS_OP_N, c, a.N, a.d_model, &one, W1 + static_cast<size_t>(s0) * a.d_model,
                     CUDA_R_16BF, a.d_model, x, CUDA_R_16BF, a.d_model, &zero, H, CUDA_R_16BF, c,
                     CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT) != CUBLAS_STATUS_SUCCESS)
      return -1;
    const long long n8 = static_cast<long long>(a.N) * c / 8;
    long long grid = (n8 + 255) / 256;
    if (grid > 8LL * num_sms) grid = 8LL * num_sms;
    relu_bf16_kernel<<<static_cast<unsigned>(grid < 1 ? 1 : grid), 256, 0, st>>>(H, n8);
    ++launches;
    // out^T [dm, N] (+)= W2_s^T [dm, c] * H^T [c, N]
    const float* beta = s0 == 0 ? &zero : &one;
    if (cublasGemmEx(b->h, CUBLAS_OP_N, CUBLAS_OP_N, a.d_model, a.N, c, &one, W2 + static_cast<size_t>(s0) * a.d_model,
                     CUDA_R_16BF, a.d_model, H, CUDA_R_16BF, c, beta, a.out, CUDA_R_32F, a.d_model,
                     CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT) != CUBLAS_STATUS_SUCCESS)
      return -1;
  }
  return cudaGetLastError() == cudaSuccess ? launches : -1;
}

}  // namespace topk
