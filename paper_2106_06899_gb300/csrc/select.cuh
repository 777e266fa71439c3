// select.cuh -- per-row streaming top-k selection, one thread per query row.
//
// The kept set of a row is the first k entries of the total order
// (score descending, key index ascending): the top-k of Eq. 4 with ties
// broken toward the lower key index.  A (score, index) pair is packed into
// one 64-bit key whose unsigned order IS that total order:
//     key = ord(score) << 32 | (~index)
// where ord() maps fp32 bit patterns to unsigned integers monotonically
// (-0 is folded onto +0 first).
//
// Each row owns a min-heap of its k best keys in shared memory, laid out
// [slot][row] so that the 32 threads of a warp always touch 32 different
// banks whatever slots they visit.  Scores stream in by ascending key index,
// so a new score can only enter when it is strictly greater than the score
// at the heap root (an equal score has a larger index and ranks lower);
// `tau` caches that root score (-inf while the heap is not yet full) and
// serves as the filter threshold.
#pragma once

#include <stdint.h>

#include "common.cuh"

namespace topk {

__device__ __forceinline__ uint32_t ord_f32(float s) {
  const uint32_t u = __float_as_uint(s + 0.0f);  // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float unord_f32(uint32_t o) {
  const uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(u);
}

__device__ __forceinline__ uint64_t make_key(float s, uint32_t j) {
  return (static_cast<uint64_t>(ord_f32(s)) << 32) | static_cast<uint64_t>(~j);
}

__device__ __forceinline__ float key_score(uint64_t key) { return unord_f32(static_cast<uint32_t>(key >> 32)); }

__device__ __forceinline__ uint32_t key_index(uint64_t key) { return ~static_cast<uint32_t>(key); }

// Exact per-row top-k (min-heap of packed keys) in shared memory.
// ROWS = number of rows sharing the [slot][row] array (the row stride).
template <int ROWS>
struct RowHeap {
  uint64_t* base;  // &heap[slot 0][this row]
  int k;           // capacity
  int n;           // entries filled
  uint64_t root;   // heap[0] once full
  float tau;       // score of heap[0] once full, else -inf

  __device__ __forceinline__ void init(uint64_t* smem, int row, int cap) {
    base = smem + row;
    k = cap;
    n = 0;
    root = 0;
    tau = -INFINITY;
  }

  __device__ __forceinline__ uint64_t get(int p) const { return base[p * ROWS]; }
  __device__ __forceinline__ void put(int p, uint64_t x) { base[p * ROWS] = x; }

  // Sift x down from slot p within a heap of m entries.
  __device__ __forceinline__ void sift_down(uint64_t x, int p, int m) {
    for (;;) {
      int c = 2 * p + 1;
      if (c >= m) break;
      uint64_t a = get(c);
      if (c + 1 < m) {
        const uint64_t b = get(c + 1);
        if (b < a) {
          a = b;
          ++c;
        }
      }
      if (a >= x) break;
      put(p, a);
      p = c;
    }
    put(p, x);
  }

  __device__ __forceinline__ void push(uint64_t x) {
    if (n < k) {
      int c = n;
      while (c > 0) {
        const int p = (c - 1) >> 1;
        const uint64_t pk = get(p);
        if (pk <= x) break;
        put(c, pk);
        c = p;
      }
      put(c, x);
      if (++n == k) {
        root = get(0);
        tau = key_score(root);
      }
    } else if (x > root) {
      sift_down(x, 0, n);
      root = get(0);
      tau = key_score(root);
    }
  }

  // Offer 32 scores whose key indices are j0 .. j0+31 (ascending).  Groups
  // of 8 are tested against tau through their maximum first; only a group
  // that beats tau is looked at element by element.
  __device__ __forceinline__ void offer32(const float (&v)[32], uint32_t j0) {
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const float m = max3f(max3f(v[8 * g], v[8 * g + 1], v[8 * g + 2]),
                            max3f(v[8 * g + 3], v[8 * g + 4], v[8 * g + 5]), fmaxf(v[8 * g + 6], v[8 * g + 7]));
      if (m > tau) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          if (v[8 * g + e] > tau) push(make_key(v[8 * g + e], j0 + 8 * g + e));
        }
      }
    }
  }

  // Heap-sort in place: afterwards slots 0 .. n-1 hold the kept keys in
  // selection order (best first).
  __device__ __forceinline__ void sort_desc() {
    if (n < k) {
      // not full: it is still a valid min-heap of n entries
    }
    for (int m = n - 1; m > 0; --m) {
      const uint64_t x = get(m);
      put(m, get(0));
      sift_down(x, 0, m);
    }
  }
};

// Replace scores of invalid keys (index >= lim) by -inf.
__device__ __forceinline__ void mask32(float (&v)[32], uint32_t j0, uint32_t lim) {
#pragma unroll
  for (int e = 0; e < 32; ++e)
    if (j0 + static_cast<uint32_t>(e) >= lim) v[e] = -INFINITY;
}

// Unpack 8 bf16 (one 16-byte vector) to fp32.
__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&f)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__device__ __forceinline__ uint4 f32x8_to_bf16(const float (&f)[8]) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    w[i] = *reinterpret_cast<uint32_t*>(&h);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Softmax over the kept entries (Eq. 4) and the weighted sum of value rows,
// for one row whose heap has been sorted.  Values are rows of D elements of
// type T (float or bf16) starting at `vbase` (row j at vbase + j * D); the
// result is written to `orow` (D elements of T).  Accumulation is fp32 over
// 64-column slices so that at most 64 accumulators are live.
template <typename T, int D, int ROWS>
__device__ __forceinline__ void softmax_gather_store(const RowHeap<ROWS>& h, const T* __restrict__ vbase,
                                                     T* __restrict__ orow) {
  constexpr int SL = D < 64 ? D : 64;
  const int n = h.n;
  const float m = n > 0 ? key_score(h.get(0)) : 0.0f;
#pragma unroll 1
  for (int c0 = 0; c0 < D; c0 += SL) {
    float acc[SL];
#pragma unroll
    for (int c = 0; c < SL; ++c) acc[c] = 0.0f;
    float z = 0.0f;
#pragma unroll 1
    for (int t = 0; t < n; ++t) {
      const uint64_t key = h.get(t);
      const float w = expf(key_score(key) - m);
      z += w;
      const T* vr = vbase + static_cast<size_t>(key_index(key)) * D + c0;
      if constexpr (sizeof(T) == 2) {
#pragma unroll
        for (int c = 0; c < SL; c += 8) {
          float f[8];
          bf16x8_to_f32(__ldg(reinterpret_cast<const uint4*>(vr + c)), f);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[c + e] = fmaf(w, f[e], acc[c + e]);
        }
      } else {
#pragma unroll
        for (int c = 0; c < SL; c += 4) {
          const float4 f = __ldg(reinterpret_cast<const float4*>(vr + c));
          acc[c] = fmaf(w, f.x, acc[c]);
          acc[c + 1] = fmaf(w, f.y, acc[c + 1]);
          acc[c + 2] = fmaf(w, f.z, acc[c + 2]);
          acc[c + 3] = fmaf(w, f.w, acc[c + 3]);
        }
      }
    }
    const float inv = n > 0 ? 1.0f / z : 0.0f;
    if constexpr (sizeof(T) == 2) {
#pragma unroll
      for (int c = 0; c < SL; c += 8) {
        float f[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) f[e] = acc[c + e] * inv;
        *reinterpret_cast<uint4*>(orow + c0 + c) = f32x8_to_bf16(f);
      }
    } else {
#pragma unroll
      for (int c = 0; c < SL; c += 4)
        *reinterpret_cast<float4*>(orow + c0 + c) =
            make_float4(acc[c] * inv, acc[c + 1] * inv, acc[c + 2] * inv, acc[c + 3] * inv);
    }
  }
}

// Debug/parity output: kept indices and fp32 scores in selection order.
template <int ROWS>
__device__ __forceinline__ void write_selection(const RowHeap<ROWS>& h, int32_t* idx_row, float* score_row) {
  for (int t = 0; t < h.k; ++t) {
    const bool have = t < h.n;
    const uint64_t key = have ? h.get(t) : 0;
    if (idx_row) idx_row[t] = have ? static_cast<int32_t>(key_index(key)) : -1;
    if (score_row) score_row[t] = have ? key_score(key) : -INFINITY;
  }
}

}  // namespace topk
