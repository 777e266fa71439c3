// attn_simt.cu -- top-k attention (Eq. 4) with scores on the CUDA cores.
//
// Serves the fp32 path (scores by sequential fp32 FMA, never TF32, as the
// paper's own fp32 runs had TF32 disabled) and the large-k path for bf16
// inputs (bf16 products are exact in fp32, accumulation fp32).  One thread
// owns one query row for the whole pass: the row's query vector sits in
// registers, key tiles of 32 rows are staged in shared memory and read by
// broadcast, and the row's top-k is kept in a shared-memory heap
// (select.cuh).  It also serves the arbitrary bit masks of Eq. 2.  After the last key tile the softmax over the k kept scores
// and the weighted sum of their value rows are written out.  No score matrix
// is stored anywhere.
#include "kernels.h"
#include "select.cuh"

namespace topk {

namespace {

constexpr int KT = 32;    // keys per staged tile
constexpr int GROUPS = 8;  // pending score groups per row

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) {
  return x;
}
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

template <typename T, int D, int ROWS>
__global__ void __launch_bounds__(ROWS) attn_simt_kernel(const T* __restrict__ q, const T* __restrict__ k,
                                                         const T* __restrict__ v, T* __restrict__ out, int BH,
                                                         int H, int Lq, int Lk, int topk, int causal,
                                                         const int32_t* __restrict__ kv_len,
                                                         const uint32_t* __restrict__ mask, long long mask_bs,
                                                         long long mask_hs, int32_t* __restrict__ idx,
                                                         float* __restrict__ score) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  float* ks = reinterpret_cast<float*>(smem_raw);                       // [KT][D]
  uint8_t* sel_mem = smem_raw + KT * D * sizeof(float);  // heap [topk][ROWS], records [GROUPS][ROWS]

  const int n_qt = (Lq + ROWS - 1) / ROWS;
  const int unit = blockIdx.x;
  // causal: heaviest query tiles first
  const int qt = causal ? (n_qt - 1 - unit / BH) : (unit % n_qt);
  const int bh = causal ? (unit % BH) : (unit / n_qt);
  const int tid = threadIdx.x;
  const int i = qt * ROWS + tid;
  const bool row_ok = i < Lq;

  float qr[D];
  {
    const T* qp = q + (static_cast<size_t>(bh) * Lq + (row_ok ? i : 0)) * D;
#pragma unroll
    for (int t = 0; t < D; ++t) qr[t] = row_ok ? to_f32(qp[t]) : 0.0f;
  }

  RowHeap<ROWS> heap;
  heap.init(sel_mem, tid, topk, GROUPS);

  // Eq. 2's masks.  Causal: the queries are the last Lq positions, key j is
  // valid for query i iff j <= i + Lk - Lq.  kv_len: the batch's key count.
  // Both give each row a valid key prefix [0, lim); the bit mask (1 = valid)
  // then removes keys anywhere in it.
  const int coff = Lk - Lq;
  const int kv_end = kv_len ? min(max(__ldg(kv_len + bh / H), 0), Lk) : Lk;
  const int kend = min(kv_end, causal ? (qt + 1) * ROWS + coff : Lk);
  const uint32_t lim = static_cast<uint32_t>(min(kv_end, causal ? min(i + 1 + coff, Lk) : Lk));
  const int cta_lim_min = min(kv_end, causal ? min(qt * ROWS + 1 + coff, Lk) : Lk);  // smallest limit here
  const T* kb = k + static_cast<size_t>(bh) * Lk * D;
  const uint32_t* mrow = nullptr;
  if (mask && row_ok)
    mrow = mask + (bh / H) * mask_bs + (bh % H) * mask_hs + static_cast<long long>(i) * ((Lk + 31) / 32);

  for (int j0 = 0; j0 < kend; j0 += KT) {
    __syncthreads();
    for (int e = tid; e < KT * D; e += ROWS) {
      const int jj = j0 + e / D;
      ks[e] = jj < Lk ? to_f32(kb[static_cast<size_t>(jj) * D + (e % D)]) : 0.0f;
    }
    __syncthreads();
    float s[KT];
#pragma unroll
    for (int e = 0; e < KT; ++e) s[e] = 0.0f;
#pragma unroll
    for (int t = 0; t < D; t += 4) {
#pragma unroll
      for (int e = 0; e < KT; ++e) {
        const float4 kv = *reinterpret_cast<const float4*>(ks + e * D + t);
        s[e] = fmaf(qr[t], kv.x, s[e]);
        s[e] = fmaf(qr[t + 1], kv.y, s[e]);
        s[e] = fmaf(qr[t + 2], kv.z, s[e]);
        s[e] = fmaf(qr[t + 3], kv.w, s[e]);
      }
    }
    if (j0 + KT > cta_lim_min) mask_scores(s, static_cast<uint32_t>(j0), lim);
    if (mask) {
      static_assert(KT == 32, "one mask word per key tile");
      const uint32_t bits = mrow ? __ldg(mrow + j0 / 32) : 0u;
#pragma unroll
      for (int e = 0; e < KT; ++e)
        if (!((bits >> e) & 1u)) s[e] = -INFINITY;
    }
    heap.offer(s, static_cast<uint32_t>(j0));
  }

  heap.finish();  // every lane takes part (warp-synchronous flush)
  if (!row_ok) return;
  const size_t orow = static_cast<size_t>(bh) * Lq + i;
  softmax_gather_store<T, D>(heap, v + static_cast<size_t>(bh) * Lk * D, out + orow * D);
  if (idx || score)
    write_selection(heap, idx ? idx + orow * topk : nullptr, score ? score + orow * topk : nullptr);
}

template <typename T, int D, int ROWS>
int launch_simt(const AttnArgs& a, cudaStream_t st) {
  const size_t smem = static_cast<size_t>(KT) * D * sizeof(float) + RowHeap<ROWS>::bytes(a.topk, GROUPS);
  auto kern = attn_simt_kernel<T, D, ROWS>;
  if (smem > 48 * 1024) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
        cudaSuccess)
      return -1;
  }
  const int BH = a.B * a.H;
  const int n_qt = (a.Lq + ROWS - 1) / ROWS;
  const long long grid = static_cast<long long>(BH) * n_qt;
  kern<<<static_cast<unsigned>(grid), ROWS, smem, st>>>(
      static_cast<const T*>(a.q), static_cast<const T*>(a.k), static_cast<const T*>(a.v), static_cast<T*>(a.out),
      BH, a.H, a.Lq, a.Lk, a.topk, a.causal, a.kv_len, a.mask, a.mask_bs, a.mask_hs, a.idx, a.score);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

}  // namespace

// Returns the number of launches (>0) on success, -1 on a CUDA error, 0 if
// the shape is not served here.
int attn_simt(const AttnArgs& a, cudaStream_t st) {
  const bool big = a.topk > kSimtSmallRowsMaxK;
  if (a.dtype == 0) {
    switch (a.d) {
      case 16: return big ? launch_simt<float, 16, 32>(a, st) : launch_simt<float, 16, 128>(a, st);
      case 32: return big ? launch_simt<float, 32, 32>(a, st) : launch_simt<float, 32, 128>(a, st);
      case 64: return big ? launch_simt<float, 64, 32>(a, st) : launch_simt<float, 64, 128>(a, st);
      case 128: return big ? launch_simt<float, 128, 32>(a, st) : launch_simt<float, 128, 128>(a, st);
      default: return 0;
    }
  }
  switch (a.d) {
    case 64: return big ? launch_simt<__nv_bfloat16, 64, 32>(a, st) : launch_simt<__nv_bfloat16, 64, 128>(a, st);
    case 128:
      return big ? launch_simt<__nv_bfloat16, 128, 32>(a, st) : launch_simt<__nv_bfloat16, 128, 128>(a, st);
    default: return 0;
  }
}

}  // namespace topk
