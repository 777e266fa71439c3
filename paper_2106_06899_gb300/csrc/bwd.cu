// bwd.cu -- backward pass of top-k attention (Eq. 4) and of the top-k
// feed-forward layer (Eq. 3) for the kept set that the forward pass cached
// (Sec. 2.2, "Improving efficiency through top-k attention").
//
// The forward pass's cache is the kept (index, score) list of every query
// row; nothing of size Lq x Lk exists at any point.  With the kept set held
// fixed, the gradient reaches q and k only through the kept scores:
//   a_t  = act(s)_t             softmax over the kept scores, or ReLU
//   da_t = dout_i . v_{j_t}
//   ds_t = a_t (da_t - sum_u a_u da_u)   (softmax)   or   da_t [s_t > 0]
//   dq_i = sum_t ds_t k_{j_t},  dk_j = sum ds_t q_i,  dv_j = sum a_t dout_i
// The last two are sums over the (i, t) that kept key j: a sparse-by-dense
// product with the pattern transposed.  Four steps:
//   1. rank:  every live entry (i, t) takes a slot in its key's bucket (an
//             atomic count per key; the count it saw is its slot);
//   2. scan:  bucket offsets, the exclusive prefix sum of the counts;
//   3. rows:  per query row the steps above up to dq_i; each entry
//             (i, ds_t, a_t, j_t) is written to its bucket slot (the FF layer
//             reads its long W1/W2 rows in column chunks, chunk-major);
//   4. keys:  the entry list, now grouped by key, is cut into equal runs of
//             entries; a lane group walks its run, adds ds q_i into dk_j and
//             a dout_i into dv_j in registers, and writes a key's sums when
//             its entries end: a plain store when the run holds all of the
//             key's entries, an atomic add when a run edge cuts them.  dk
//             and dv are zeroed first, so keys that no row kept read 0.
// Every run of entries is the same length whatever the keys' popularity,
// so a key that many rows keep does not serialise one warp.  The order in
// which a key's terms are added depends on the atomic ranks: results can
// differ in the last bits from call to call.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.h"

namespace topk {

namespace {

struct __align__(16) BwdEntry {
  int row;   // global query row (b, h, i) flattened, or token
  float ds;  // dL/ds_t
  float a;   // a_t
  int key;   // bucket: (b, h) flattened times Lk plus the key index j
};

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}

// 16 bytes of T widened to floats (bf16 -> f32 is exact: a 16-bit shift)
template <typename T>
struct Chunk;
template <>
struct Chunk<__nv_bfloat16> {
  static constexpr int N = 8;
  __device__ __forceinline__ static void load(const __nv_bfloat16* p, float (&f)[8]) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
};
template <>
struct Chunk<float> {
  static constexpr int N = 4;
  __device__ __forceinline__ static void load(const float* p, float (&f)[4]) {
    const float4 u = __ldg(reinterpret_cast<const float4*>(p));
    f[0] = u.x;
    f[1] = u.y;
    f[2] = u.z;
    f[3] = u.w;
  }
};

// n floats of a row that starts 16-byte aligned, as float4 loads
template <int N>
__device__ __forceinline__ void load_f32(const float* p, float (&f)[N]) {
#pragma unroll
  for (int i = 0; i < N / 4; ++i) {
    const float4 u = __ldg(reinterpret_cast<const float4*>(p) + i);
    f[4 * i] = u.x;
    f[4 * i + 1] = u.y;
    f[4 * i + 2] = u.z;
    f[4 * i + 3] = u.w;
  }
}

// the same columns of a dout row, which may be bf16 or fp32
template <typename TD, int N>
__device__ __forceinline__ void load_cols(const TD* p, float (&f)[N]) {
  if constexpr (sizeof(TD) == 4) {
    load_f32<N>(reinterpret_cast<const float*>(p), f);
  } else {
    static_assert(N % 8 == 0, "bf16 columns come in 16-byte chunks");
#pragma unroll
    for (int i = 0; i < N / 8; ++i) {
      float g[8];
      Chunk<__nv_bfloat16>::load(reinterpret_cast<const __nv_bfloat16*>(p) + 8 * i, g);
#pragma unroll
      for (int e = 0; e < 8; ++e) f[8 * i + e] = g[e];
    }
  }
}

// ---------------------------------------------------------------------------
// 1. rank
__global__ void bwd_rank_kernel(const int32_t* __restrict__ idx, const float* __restrict__ score,
                                long long n_entries, int K, int Lq, int Lk, int relu, int* __restrict__ cnt,
                                int* __restrict__ rank) {
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  for (long long e = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; e < n_entries; e += stride) {
    const int j = idx[e];
    int r = -1;
    // an empty slot (-1), and under ReLU a kept score <= 0 (a_t = ds_t = 0),
    // contributes nothing
    if (j >= 0 && j < Lk && !(relu && !(score[e] > 0.f))) {
      const long long bh = e / K / Lq;
      r = atomicAdd(&cnt[bh * Lk + j], 1);
    }
    rank[e] = r;
  }
}

// ---------------------------------------------------------------------------
// 2. scan: tiles of 4096 counts, 1024 threads x 4
constexpr int kScanThreads = 1024;
constexpr int kScanTile = 4096;

// exclusive prefix of v over the block; *total gets the block's sum
__device__ __forceinline__ int block_exclusive_scan(int v, int* total) {
  __shared__ int ws[32];
  __shared__ int tot;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) ws[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < (blockDim.x >> 5) ? ws[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += y;
    }
    ws[lane] = wi - w;  // exclusive prefix of the warp sums
    if (lane == 31) tot = wi;
  }
  __syncthreads();
  const int res = ws[warp] + incl - v;
  *total = tot;
  __syncthreads();
  return res;
}

__global__ void __launch_bounds__(kScanThreads) scan_tile_sums_kernel(const int* __restrict__ cnt, long long n,
                                                                      int* __restrict__ bsum) {
  const long long base = static_cast<long long>(blockIdx.x) * kScanTile + threadIdx.x * 4;
  int s = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    if (base + i < n) s += cnt[base + i];
  int total;
  block_exclusive_scan(s, &total);
  if (threadIdx.x == 0) bsum[blockIdx.x] = total;
}

// one block: exclusive scan of the nb tile sums in place; off[n] = total
__global__ void __launch_bounds__(kScanThreads) scan_tile_offsets_kernel(int* __restrict__ bsum, int nb,
                                                                         int* __restrict__ off, long long n) {
  int carry = 0;
  for (int b0 = 0; b0 < nb; b0 += kScanThreads) {
    const int b = b0 + threadIdx.x;
    const int v = b < nb ? bsum[b] : 0;
    int total;
    const int ex = block_exclusive_scan(v, &total);
    if (b < nb) bsum[b] = carry + ex;
    carry += total;
  }
  if (threadIdx.x == 0) off[n] = carry;
}

__global__ void __launch_bounds__(kScanThreads) scan_apply_kernel(const int* __restrict__ cnt, long long n,
                                                                  const int* __restrict__ bsum, int* __restrict__ off) {
  const long long base = static_cast<long long>(blockIdx.x) * kScanTile + threadIdx.x * 4;
  int v[4], s = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[i] = base + i < n ? cnt[base + i] : 0;
    s += v[i];
  }
  int total;
  int ex = block_exclusive_scan(s, &total) + bsum[blockIdx.x];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (base + i < n) off[base + i] = ex;
    ex += v[i];
  }
}

// ---------------------------------------------------------------------------
// 3a. rows, softmax attention.  One warp per query row; a group of LPR lanes
// reads one key/value row (one 16-byte chunk per lane), G = 32 / LPR rows per
// step.  Per warp, shared memory holds a_t and then ds_t for the row's K
// entries.
constexpr int kRowWarps = 8;

template <typename T, int D>
__global__ void __launch_bounds__(kRowWarps * 32) attn_bwd_rows_kernel(
    const T* __restrict__ k, const T* __restrict__ v, const T* __restrict__ dout, const int32_t* __restrict__ idx,
    const float* __restrict__ score, const int* __restrict__ rank, const int* __restrict__ off,
    BwdEntry* __restrict__ ent, float* __restrict__ dq, long long R, int Lq, int Lk, int K) {
  constexpr int VEC = Chunk<T>::N;
  constexpr int LPR = D / VEC;
  constexpr int G = 32 / LPR;
  static_assert(LPR >= 1 && LPR <= 32 && 32 % LPR == 0, "a key row spans 1..32 lanes");
  extern __shared__ float sm[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* pa = sm + static_cast<size_t>(warp) * 2 * K;
  float* pg = pa + K;
  const int grp = lane / LPR, c = lane % LPR;
  for (long long row = static_cast<long long>(blockIdx.x) * kRowWarps + warp; row < R;
       row += static_cast<long long>(gridDim.x) * kRowWarps) {
    const long long bh = row / Lq;
    const int32_t* ki = idx + row * K;
    const float* ks = score + row * K;
    // softmax over the kept scores (Eq. 4), recomputed from the cache
    float m = -INFINITY;
    for (int t = lane; t < K; t += 32) {
      const int j = ki[t];
      if (j >= 0 && j < Lk) m = fmaxf(m, ks[t]);
    }
    m = warp_max(m);
    float z = 0.f;
    for (int t = lane; t < K; t += 32) {
      const int j = ki[t];
      const float e = (j >= 0 && j < Lk) ? expf(ks[t] - m) : 0.f;
      pa[t] = e;
      z += e;
    }
    z = warp_sum(z);
    const float inv = z > 0.f ? 1.f / z : 0.f;
    // da_t = dout_i . v_{j_t}
    float go[VEC];
    Chunk<T>::load(dout + row * D + c * VEC, go);
    const T* vb = v + bh * Lk * D + c * VEC;
    const T* kb = k + bh * Lk * D + c * VEC;
#pragma unroll 4
    for (int t0 = 0; t0 < K; t0 += G) {
      const int t = t0 + grp;
      const int j = t < K ? ki[t] : -1;
      float p = 0.f;
      if (j >= 0 && j < Lk) {
        float f[VEC];
        Chunk<T>::load(vb + static_cast<long long>(j) * D, f);
#pragma unroll
        for (int e = 0; e < VEC; ++e) p = fmaf(f[e], go[e], p);
      }
#pragma unroll
      for (int o = LPR / 2; o > 0; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
      if (c == 0 && t < K) pg[t] = p;
    }
    __syncwarp();
    // ds_t = a_t (da_t - sum_u a_u da_u)
    float dot = 0.f;
    for (int t = lane; t < K; t += 32) dot = fmaf(pa[t] * inv, pg[t], dot);
    dot = warp_sum(dot);
    for (int t = lane; t < K; t += 32) {
      const float a = pa[t] * inv;
      pg[t] = a * (pg[t] - dot);
      pa[t] = a;
    }
    __syncwarp();
    // dq_i = sum_t ds_t k_{j_t}
    float acc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e) acc[e] = 0.f;
#pragma unroll 4
    for (int t0 = 0; t0 < K; t0 += G) {
      const int t = t0 + grp;
      const int j = t < K ? ki[t] : -1;
      if (j >= 0 && j < Lk) {
        float f[VEC];
        Chunk<T>::load(kb + static_cast<long long>(j) * D, f);
        const float g = pg[t];
#pragma unroll
        for (int e = 0; e < VEC; ++e) acc[e] = fmaf(g, f[e], acc[e]);
      }
    }
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
      for (int e = 0; e < VEC; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    if (grp == 0) {
      float4* dst = reinterpret_cast<float4*>(dq + row * D + c * VEC);
#pragma unroll
      for (int e = 0; e < VEC / 4; ++e) dst[e] = make_float4(acc[4 * e], acc[4 * e + 1], acc[4 * e + 2], acc[4 * e + 3]);
    }
    // the entries go to their keys' buckets
    for (int t = lane; t < K; t += 32) {
      const int r = rank[row * K + t];
      if (r >= 0) {
        const int j = ki[t];
        BwdEntry en;
        en.row = static_cast<int>(row);
        en.ds = pg[t];
        en.a = pa[t];
        en.key = static_cast<int>(bh * Lk + j);
        ent[off[bh * Lk + j] + r] = en;
      }
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------
// 3b. rows, the ReLU feed-forward layer, in column chunks of kFfChunk.  A
// token's k rows of W2 (and of W1) are 2 KB each at d_model = 1024 and W1 and
// W2 together exceed L2, so the rows are read chunk-major: all tokens read
// their rows' first kFfChunk columns before any reads the next chunk, and the
// columns in use (d_ff x kFfChunk bf16, 32 MB at d_ff = 65536) stay in L2.
//   da:  per (chunk, token) a warp per kept entry sums dout_i . W2_j over the
//        chunk's columns (one 16-byte vector per lane, a warp sum) into
//        part[chunk][token][t];
//   dx:  per (chunk, token) ds_t = sum over chunks of part (0 unless s_t > 0,
//        ReLU's backward), then dx_i = sum_t ds_t W1_{j_t} over the chunk's
//        columns (each thread 4 columns, 8 rows in flight); the chunk-0 CTA
//        of a token also writes its entries to their key buckets.
constexpr int kFfChunk = 256;
constexpr int kDaWarps = 8;
constexpr int kDxThreads = kFfChunk / 4;

__global__ void __launch_bounds__(kDaWarps * 32) ffn_bwd_da_kernel(
    const __nv_bfloat16* __restrict__ W2, const float* __restrict__ dout, const int32_t* __restrict__ idx,
    const float* __restrict__ score, float* __restrict__ part, int N, int DM, int dff, int K) {
  const int i = blockIdx.x % N, chunk = blockIdx.x / N;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int col = chunk * kFfChunk + lane * 8;
  const bool live = col < DM;
  float g[8];
  if (live)
    load_f32<8>(dout + static_cast<long long>(i) * DM + col, g);
  else
#pragma unroll
    for (int e = 0; e < 8; ++e) g[e] = 0.f;
  const int32_t* ki = idx + static_cast<long long>(i) * K;
  const float* ks = score + static_cast<long long>(i) * K;
  float* out = part + (static_cast<long long>(chunk) * N + i) * K;
  constexpr int U = 4;  // kept entries in flight per warp
  for (int t0 = warp * U; t0 < K; t0 += kDaWarps * U) {
    float f[U][8];
    bool use[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = t0 + u;
      const int j = t < K ? ki[t] : -1;
      use[u] = t < K && j >= 0 && j < dff && ks[t] > 0.f;
      if (use[u] && live)
        Chunk<__nv_bfloat16>::load(W2 + static_cast<long long>(j) * DM + col, f[u]);
      else
#pragma unroll
        for (int e = 0; e < 8; ++e) f[u][e] = 0.f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float p = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) p = fmaf(f[u][e], g[e], p);
      p = warp_sum(p);
      if (lane == 0 && t0 + u < K) out[t0 + u] = use[u] ? p : 0.f;
    }
  }
}

__global__ void __launch_bounds__(kDxThreads) ffn_bwd_dx_kernel(
    const __nv_bfloat16* __restrict__ W1, const int32_t* __restrict__ idx, const float* __restrict__ score,
    const float* __restrict__ part, const int* __restrict__ rank, const int* __restrict__ off,
    BwdEntry* __restrict__ ent, float* __restrict__ dx, int N, int DM, int dff, int K, int nchunks) {
  extern __shared__ float dsv[];  // [K] ds_t, then [K] key indices (as int)
  int* jv = reinterpret_cast<int*>(dsv + K);
  const int i = blockIdx.x % N, chunk = blockIdx.x / N;
  const int tid = threadIdx.x;
  for (int t = tid; t < K; t += kDxThreads) {
    const int j = idx[static_cast<long long>(i) * K + t];
    const float s = score[static_cast<long long>(i) * K + t];
    const bool use = j >= 0 && j < dff && s > 0.f;
    float ds = 0.f;
    if (use)
      for (int c = 0; c < nchunks; ++c) ds += part[(static_cast<long long>(c) * N + i) * K + t];
    dsv[t] = ds;
    jv[t] = use ? j : -1;
    if (chunk == 0 && use) {  // this token's entries go to their key buckets once
      BwdEntry en;
      en.row = i;
      en.ds = ds;
      en.a = s;
      en.key = j;
      ent[off[j] + rank[static_cast<long long>(i) * K + t]] = en;
    }
  }
  __syncthreads();
  const int c0 = chunk * kFfChunk + tid * 4;
  if (c0 >= DM) return;
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  for (int t0 = 0; t0 < K; t0 += 8) {
    uint2 raw[8];
    float w[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int t = t0 + u;
      const int j = t < K ? jv[t] : -1;
      w[u] = j >= 0 ? dsv[t] : 0.f;
      raw[u] = j >= 0 ? __ldg(reinterpret_cast<const uint2*>(W1 + static_cast<long long>(j) * DM + c0))
                      : make_uint2(0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      a0 = fmaf(w[u], __uint_as_float(raw[u].x << 16), a0);
      a1 = fmaf(w[u], __uint_as_float(raw[u].x & 0xffff0000u), a1);
      a2 = fmaf(w[u], __uint_as_float(raw[u].y << 16), a2);
      a3 = fmaf(w[u], __uint_as_float(raw[u].y & 0xffff0000u), a3);
    }
  }
  *reinterpret_cast<float4*>(dx + static_cast<long long>(i) * DM + c0) = make_float4(a0, a1, a2, a3);
}

// ---------------------------------------------------------------------------
// 4. keys.  The entry list is grouped by bucket (one bucket per key of each
// (b, h)).  Lane groups of LPR lanes each take a run of kRun consecutive
// entries; lane c of a group covers the 16-byte chunks c, c + LPR, ... (CPL
// of them) of a q (or x) row and the same columns of dout, within the column
// slice of its grid row (blockIdx.y; the FF layer's 2 KB rows are split into
// 256-column slices).  A bucket's sums
// are written when its entries end inside the run: stored when the run
// holds all of them, added atomically when they continue past either end of
// the run.  U entries are loaded ahead so that their row reads overlap.
constexpr int kKeyWarps = 8;
constexpr int kRun = 64;

template <typename T, typename TD, int LPR, int CPL>
__global__ void __launch_bounds__(kKeyWarps * 32) bwd_keys_kernel(
    const T* __restrict__ q, const TD* __restrict__ dout, const BwdEntry* __restrict__ ent,
    const int* __restrict__ total_ptr, float* __restrict__ dk, float* __restrict__ dv, int D) {
  constexpr int VEC = Chunk<T>::N;
  constexpr int G = 32 / LPR;
  constexpr int U = CPL >= 4 ? 1 : 4 / CPL;
  static_assert(LPR >= 1 && LPR <= 32 && 32 % LPR == 0, "a row spans 1..32 lanes of a group");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane / LPR, c = lane % LPR;
  const int nch = D / VEC;
  const int ch0 = blockIdx.y * LPR * CPL;  // the column slice of this grid row
  const long long E = *total_ptr;
  const long long n_runs = (E + kRun - 1) / kRun;
  const long long stride = static_cast<long long>(gridDim.x) * kKeyWarps * G;
  for (long long run = (static_cast<long long>(blockIdx.x) * kKeyWarps + warp) * G + grp; run < n_runs;
       run += stride) {
    const long long s0 = run * kRun;
    const long long s1 = s0 + kRun < E ? s0 + kRun : E;
    float ak[CPL][VEC], av[CPL][VEC];
#pragma unroll
    for (int u = 0; u < CPL; ++u)
#pragma unroll
      for (int e = 0; e < VEC; ++e) ak[u][e] = av[u][e] = 0.f;
    int cur = ent[s0].key;
    bool head_cut = s0 > 0 && ent[s0 - 1].key == cur;  // its entries began before this run
    auto flush = [&](bool partial) {
#pragma unroll
      for (int u = 0; u < CPL; ++u) {
        const int ch = ch0 + c + LPR * u;
        if (ch < nch) {
          float4* pk = reinterpret_cast<float4*>(dk + static_cast<long long>(cur) * D + ch * VEC);
          float4* pv = reinterpret_cast<float4*>(dv + static_cast<long long>(cur) * D + ch * VEC);
#pragma unroll
          for (int e = 0; e < VEC / 4; ++e) {
            const float4 xk = make_float4(ak[u][4 * e], ak[u][4 * e + 1], ak[u][4 * e + 2], ak[u][4 * e + 3]);
            const float4 xv = make_float4(av[u][4 * e], av[u][4 * e + 1], av[u][4 * e + 2], av[u][4 * e + 3]);
            if (partial) {
              atomicAdd(pk + e, xk);
              atomicAdd(pv + e, xv);
            } else {
              pk[e] = xk;
              pv[e] = xv;
            }
          }
        }
#pragma unroll
        for (int e = 0; e < VEC; ++e) ak[u][e] = av[u][e] = 0.f;
      }
    };
    for (long long e0 = s0; e0 < s1; e0 += U) {
      BwdEntry en[U];
      float fq[U][CPL][VEC], fg[U][CPL][VEC];
#pragma unroll
      for (int i = 0; i < U; ++i) {
        const bool ok = e0 + i < s1;
        en[i] = ok ? ent[e0 + i] : BwdEntry{0, 0.f, 0.f, -1};
#pragma unroll
        for (int u = 0; u < CPL; ++u) {
          const int ch = ch0 + c + LPR * u;
          if (ok && ch < nch) {
            Chunk<T>::load(q + static_cast<long long>(en[i].row) * D + ch * VEC, fq[i][u]);
            load_cols<TD, VEC>(dout + static_cast<long long>(en[i].row) * D + ch * VEC, fg[i][u]);
          } else {
#pragma unroll
            for (int e = 0; e < VEC; ++e) fq[i][u][e] = fg[i][u][e] = 0.f;
          }
        }
      }
#pragma unroll
      for (int i = 0; i < U; ++i) {
        if (e0 + i >= s1) break;
        if (en[i].key != cur) {  // cur's entries ended inside this run
          flush(head_cut);
          cur = en[i].key;
          head_cut = false;
        }
#pragma unroll
        for (int u = 0; u < CPL; ++u)
#pragma unroll
          for (int e = 0; e < VEC; ++e) {
            ak[u][e] = fmaf(en[i].ds, fq[i][u][e], ak[u][e]);
            av[u][e] = fmaf(en[i].a, fg[i][u][e], av[u][e]);
          }
      }
    }
    const bool tail_cut = s1 < E && ent[s1].key == cur;
    flush(head_cut || tail_cut);
  }
}

// ---------------------------------------------------------------------------
// launchers

int grid_for(long long items, int per_block, int num_sms, int blocks_per_sm) {
  long long g = (items + per_block - 1) / per_block;
  const long long cap = static_cast<long long>(num_sms) * blocks_per_sm;
  if (g > cap) g = cap;
  return static_cast<int>(g < 1 ? 1 : g);
}

// Workspace layout (each part 256-byte aligned): cnt [nb], off [nb + 1],
// tile sums [ceil(nb / 4096)], rank [E], entries [E] (E = rows x K).
struct BwdScratch {
  int* cnt;
  int* off;
  int* bsum;
  int* rank;
  BwdEntry* ent;
  float* part;  // FF only: per column chunk, token and kept entry, the partial dout . W2_j
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t scratch_bytes(long long n_buckets, long long n_entries, long long n_part = 0) {
  const long long n_tiles = (n_buckets + kScanTile - 1) / kScanTile;
  return align256(n_buckets * 4) + align256((n_buckets + 1) * 4) + align256(n_tiles * 4) +
         align256(n_entries * 4) + align256(n_entries * sizeof(BwdEntry)) + align256(n_part * 4);
}

BwdScratch carve(void* ws, long long n_buckets, long long n_entries) {
  const long long n_tiles = (n_buckets + kScanTile - 1) / kScanTile;
  uint8_t* p = static_cast<uint8_t*>(ws);
  BwdScratch s;
  s.cnt = reinterpret_cast<int*>(p);
  p += align256(n_buckets * 4);
  s.off = reinterpret_cast<int*>(p);
  p += align256((n_buckets + 1) * 4);
  s.bsum = reinterpret_cast<int*>(p);
  p += align256(n_tiles * 4);
  s.rank = reinterpret_cast<int*>(p);
  p += align256(n_entries * 4);
  s.ent = reinterpret_cast<BwdEntry*>(p);
  p += align256(n_entries * sizeof(BwdEntry));
  s.part = reinterpret_cast<float*>(p);
  return s;
}

// steps 1 and 2; returns the number of launches, -1 on a CUDA error
int rank_and_scan(const BwdScratch& s, const int32_t* idx, const float* score, long long n_entries, int K, int Lq,
                  int Lk, long long n_buckets, int relu, int num_sms, cudaStream_t st) {
  if (cudaMemsetAsync(s.cnt, 0, n_buckets * 4, st) != cudaSuccess) return -1;
  bwd_rank_kernel<<<grid_for(n_entries, 256, num_sms, 8), 256, 0, st>>>(idx, score, n_entries, K, Lq, Lk, relu,
                                                                       s.cnt, s.rank);
  const long long n_tiles = (n_buckets + kScanTile - 1) / kScanTile;
  scan_tile_sums_kernel<<<static_cast<unsigned>(n_tiles), kScanThreads, 0, st>>>(s.cnt, n_buckets, s.bsum);
  scan_tile_offsets_kernel<<<1, kScanThreads, 0, st>>>(s.bsum, static_cast<int>(n_tiles), s.off, n_buckets);
  scan_apply_kernel<<<static_cast<unsigned>(n_tiles), kScanThreads, 0, st>>>(s.cnt, n_buckets, s.bsum, s.off);
  return cudaGetLastError() == cudaSuccess ? 4 : -1;
}

// slices > 1 splits each row into column slices of LPR * CPL 16-byte chunks,
// one grid row per slice: lighter lane groups, more of them in flight
template <typename T, typename TD, int LPR, int CPL>
int launch_keys(const T* q, const TD* dout, const BwdScratch& s, long long n_buckets, long long max_entries,
                float* dk, float* dv, int D, int num_sms, cudaStream_t st, int slices = 1) {
  constexpr int G = 32 / LPR;
  const long long runs = (max_entries + kRun - 1) / kRun;
  const dim3 grid(grid_for(runs, kKeyWarps * G, num_sms, 8), slices);
  bwd_keys_kernel<T, TD, LPR, CPL><<<grid, kKeyWarps * 32, 0, st>>>(q, dout, s.ent, s.off + n_buckets, dk, dv, D);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

template <typename T, int D>
int attn_bwd_t(const AttnBwdArgs& a, int num_sms, cudaStream_t st) {
  constexpr int VEC = Chunk<T>::N;
  constexpr int LPR = D / VEC;
  const long long R = static_cast<long long>(a.B) * a.H * a.Lq;
  const long long n_entries = R * a.topk;
  const long long n_buckets = static_cast<long long>(a.B) * a.H * a.Lk;
  const BwdScratch s = carve(a.workspace, n_buckets, n_entries);
  const T* q = static_cast<const T*>(a.q);
  const T* k = static_cast<const T*>(a.k);
  const T* v = static_cast<const T*>(a.v);
  const T* g = static_cast<const T*>(a.dout);
  const size_t kv_bytes = static_cast<size_t>(n_buckets) * D * sizeof(float);
  if (cudaMemsetAsync(a.dk, 0, kv_bytes, st) != cudaSuccess || cudaMemsetAsync(a.dv, 0, kv_bytes, st) != cudaSuccess)
    return -1;
  int n = rank_and_scan(s, a.idx, a.score, n_entries, a.topk, a.Lq, a.Lk, n_buckets, 0, num_sms, st);
  if (n < 0) return -1;
  const size_t smem = static_cast<size_t>(kRowWarps) * 2 * a.topk * sizeof(float);
  auto rows = attn_bwd_rows_kernel<T, D>;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(rows, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
    return -1;
  rows<<<grid_for(R, kRowWarps, num_sms, 8), kRowWarps * 32, smem, st>>>(k, v, g, a.idx, a.score, s.rank, s.off,
                                                                          s.ent, a.dq, R, a.Lq, a.Lk, a.topk);
  if (cudaGetLastError() != cudaSuccess) return -1;
  n += 1;
  const int nk = launch_keys<T, T, LPR, 1>(q, g, s, n_buckets, n_entries, a.dk, a.dv, D, num_sms, st);
  return nk < 0 ? -1 : n + nk;
}

int ffn_bwd_t(const FfnBwdArgs& a, int num_sms, cudaStream_t st) {
  const long long n_entries = static_cast<long long>(a.N) * a.topk;
  const long long n_buckets = a.d_ff;
  const BwdScratch s = carve(a.workspace, n_buckets, n_entries);
  const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(a.x);
  const __nv_bfloat16* W1 = static_cast<const __nv_bfloat16*>(a.W1);
  const __nv_bfloat16* W2 = static_cast<const __nv_bfloat16*>(a.W2);
  const size_t w_bytes = static_cast<size_t>(a.d_ff) * a.d_model * sizeof(float);
  if (cudaMemsetAsync(a.dW1, 0, w_bytes, st) != cudaSuccess || cudaMemsetAsync(a.dW2, 0, w_bytes, st) != cudaSuccess)
    return -1;
  int n = rank_and_scan(s, a.idx, a.score, n_entries, a.topk, a.N, a.d_ff, n_buckets, 1, num_sms, st);
  if (n < 0) return -1;
  const int nchunks = (a.d_model + kFfChunk - 1) / kFfChunk;
  const unsigned grid = static_cast<unsigned>(nchunks) * static_cast<unsigned>(a.N);
  ffn_bwd_da_kernel<<<grid, kDaWarps * 32, 0, st>>>(W2, a.dout, a.idx, a.score, s.part, a.N, a.d_model, a.d_ff,
                                                    a.topk);
  const size_t smem = static_cast<size_t>(a.topk) * 8;
  ffn_bwd_dx_kernel<<<grid, kDxThreads, smem, st>>>(W1, a.idx, a.score, s.part, s.rank, s.off, s.ent, a.dx, a.N,
                                                    a.d_model, a.d_ff, a.topk, nchunks);
  if (cudaGetLastError() != cudaSuccess) return -1;
  n += 2;
  const int nk = launch_keys<__nv_bfloat16, float, 32, 1>(x, a.dout, s, n_buckets, n_entries, a.dW1, a.dW2,
                                                           a.d_model, num_sms, st, nchunks);
  return nk < 0 ? -1 : n + nk;
}

}  // namespace

size_t attn_bwd_workspace_bytes(int B, int H, int Lq, int Lk, int topk) {
  const long long R = static_cast<long long>(B) * H * Lq;
  return scratch_bytes(static_cast<long long>(B) * H * Lk, R * topk);
}

size_t ffn_bwd_workspace_bytes(int N, int d_model, int d_ff, int topk) {
  const long long nchunks = (d_model + kFfChunk - 1) / kFfChunk;
  return scratch_bytes(d_ff, static_cast<long long>(N) * topk, nchunks * N * topk);
}

bool attn_bwd_supports(int d, int dtype) {
  if (dtype == 1) return d == 64 || d == 128;
  return d == 16 || d == 32 || d == 64 || d == 128;
}

int attn_bwd(const AttnBwdArgs& a, int num_sms, cudaStream_t st) {
  if (a.dtype == 1) {
    if (a.d == 64) return attn_bwd_t<__nv_bfloat16, 64>(a, num_sms, st);
    if (a.d == 128) return attn_bwd_t<__nv_bfloat16, 128>(a, num_sms, st);
    return 0;
  }
  switch (a.d) {
    case 16: return attn_bwd_t<float, 16>(a, num_sms, st);
    case 32: return attn_bwd_t<float, 32>(a, num_sms, st);
    case 64: return attn_bwd_t<float, 64>(a, num_sms, st);
    case 128: return attn_bwd_t<float, 128>(a, num_sms, st);
    default: return 0;
  }
}

int ffn_bwd(const FfnBwdArgs& a, int num_sms, cudaStream_t st) {
  return ffn_bwd_t(a, num_sms, st);
}

}  // namespace topk
