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
// banks whatever slots they visit (128 rows: a 64-bit slot row is 1 KB).  Scores stream in by ascending key index,
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

// Exact per-row top-k: a 4-ary min-heap of packed keys in shared memory,
// fed through a per-row buffer of pending score groups.
//
// The filter compares the maximum of each group of 8 scores with tau (the
// heap root's score, -inf until the heap is full) and, if it wins, copies
// the whole group (8 scores and its first key index) into the row's record
// buffer with two vector stores: no per-element work and no loop on the
// divergent path.  When any lane of the warp has filled its record buffer,
// the whole warp expands its records into the heaps in lockstep (flush):
// elements are offered in ascending key index, each one that beats the
// current root replaces it.  tau only rises, so records taken against a
// stale tau can hold a few elements that no longer qualify; they are
// re-checked at expansion.  The 4-ary heap halves the dependent shared
// memory round trips of a replace (log4 k levels of four independent loads).
// ROWS = number of rows sharing the [slot][row] arrays (the row stride);
// every call of offer*/flush/finish must be made by all 32 lanes of a warp.
template <int ROWS, int FIXED_K = 0>
struct RowHeap {
  // FIXED_K == 64: an 8-ary heap of exactly 64 keys, padded with 9 sentinel
  // slots (largest key) so that every interior node has 8 children: a root
  // replacement is two fully unrolled levels of 8 independent loads.
  static constexpr int kPad = FIXED_K == 64 ? 9 : 0;
  uint64_t* base;  // &heap[slot 0][this row]
  float4* rlo;     // &records_lo[0][this row]: scores 0..3
  float4* rhi;     // &records_hi[0][this row]: scores 4..7
  uint32_t* rj;    // &records_j0[0][this row]
  uint8_t* stage;  // &stage[0][this row]: codes (record slot * 8 + element) of elements to offer
  int k;           // capacity
  int n;           // entries filled
  int rc;          // records pending
  int gr;          // record capacity
  uint64_t root;   // heap[0] once full
  float tau;       // score of heap[0] once full, else -inf

  // shared memory: heap (k + kPad) x ROWS x 8 bytes, records (gr + 1) x ROWS
  // x 36 bytes (the last one a scratch slot), stage 8 gr x ROWS bytes (gr <=
  // 31, so that a code fits in one byte)
  __host__ __device__ static constexpr size_t bytes(int k_, int gr_) {
    return static_cast<size_t>(ROWS) *
           (static_cast<size_t>(k_ + kPad) * 8 + static_cast<size_t>(gr_ + 1) * 36 + static_cast<size_t>(gr_) * 8);
  }

  __device__ __forceinline__ void init(uint8_t* smem, int row, int cap, int rec_cap) {
    base = reinterpret_cast<uint64_t*>(smem) + row;
    uint8_t* r = smem + static_cast<size_t>(cap + kPad) * ROWS * 8;
    for (int q = 0; q < kPad; ++q) base[(cap + q) * ROWS] = ~0ull;  // sentinels never leave the leaves
    const size_t nrec = static_cast<size_t>(rec_cap) + 1;  // + scratch slot
    rlo = reinterpret_cast<float4*>(r) + row;
    rhi = reinterpret_cast<float4*>(r + nrec * ROWS * 16) + row;
    rj = reinterpret_cast<uint32_t*>(r + nrec * ROWS * 32) + row;
    stage = r + nrec * ROWS * 36 + row;
    k = cap;
    gr = rec_cap;
    n = 0;
    rc = 0;
    root = 0;
    tau = -INFINITY;
  }

  __device__ __forceinline__ uint64_t get(int p) const { return base[p * ROWS]; }
  __device__ __forceinline__ void put(int p, uint64_t x) { base[p * ROWS] = x; }

  // Sift x down from slot p within a heap of m entries (children 4p+1..4p+4).
  __device__ __forceinline__ void sift_down(uint64_t x, int p, int m) {
    for (;;) {
      const int c = 4 * p + 1;
      if (c >= m) break;
      uint64_t a = get(c);
      int ca = c;
      if (c + 3 < m) {
        const uint64_t b1 = get(c + 1), b2 = get(c + 2), b3 = get(c + 3);
        const uint64_t m01 = b1 < a ? b1 : a;
        const int i01 = b1 < a ? c + 1 : c;
        const uint64_t m23 = b3 < b2 ? b3 : b2;
        const int i23 = b3 < b2 ? c + 3 : c + 2;
        a = m23 < m01 ? m23 : m01;
        ca = m23 < m01 ? i23 : i01;
      } else {
        for (int q = c + 1; q < m; ++q) {
          const uint64_t b = get(q);
          if (b < a) {
            a = b;
            ca = q;
          }
        }
      }
      if (a >= x) break;
      put(p, a);
      p = ca;
    }
    put(p, x);
  }

  // 8-ary heap of 64 keys: children of node p are 8p+1 .. 8p+8; slots 64..72
  // hold sentinels.  Replace the root by x and restore the heap order.
  __device__ __forceinline__ void replace_root64(uint64_t x) {
    int p = 0;
    bool done = false;
#pragma unroll
    for (int level = 0; level < 2; ++level) {
      const int c = 8 * p + 1;
      uint64_t ch[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) ch[q] = get(c + q);
      // argmin over 8 keys, tree of depth 3
      uint64_t m2[4];
      int i2[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const bool lo = ch[2 * q] <= ch[2 * q + 1];
        m2[q] = lo ? ch[2 * q] : ch[2 * q + 1];
        i2[q] = lo ? 2 * q : 2 * q + 1;
      }
      const bool l01 = m2[0] <= m2[1], l23 = m2[2] <= m2[3];
      const uint64_t m01 = l01 ? m2[0] : m2[1], m23 = l23 ? m2[2] : m2[3];
      const int i01 = l01 ? i2[0] : i2[1], i23 = l23 ? i2[2] : i2[3];
      const bool lf = m01 <= m23;
      const uint64_t a = lf ? m01 : m23;
      const int ca = c + (lf ? i01 : i23);
      if (!done && a < x) {
        put(p, a);
        p = ca;
      } else {
        done = true;
      }
    }
    put(p, x);
  }

  // Add x: while the heap is not full it is appended (the heap is built
  // once, when the k-th entry arrives); afterwards it replaces the root if it
  // ranks above it.
  __device__ __forceinline__ void push(uint64_t x) {
    if (n < k) {
      put(n, x);
      if (++n == k) {
        if constexpr (FIXED_K == 64) {
          // build the 8-ary heap: nodes 8..1 (level 1), then the root
          for (int p = 8; p >= 1; --p) sift_down8(get(p), p);
          sift_down8(get(0), 0);
        } else {
          for (int p = (k - 2) / 4; p >= 0; --p) sift_down(get(p), p, k);
        }
        root = get(0);
        tau = key_score(root);
      }
    } else if (x > root) {
      if constexpr (FIXED_K == 64) {
        replace_root64(x);
      } else {
        sift_down(x, 0, k);
      }
      root = get(0);
      tau = key_score(root);
    }
  }

  // Sift down in the 8-ary heap of 64 (used to build it and to sort it).
  // m: number of live entries (slots >= m are treated as absent).
  __device__ __forceinline__ void sift_down8(uint64_t x, int p, int m = 64) {
    for (;;) {
      const int c = 8 * p + 1;
      if (c >= m) break;
      uint64_t a = get(c);
      int ca = c;
      for (int q = c + 1; q < c + 8 && q < m; ++q) {
        const uint64_t b = get(q);
        if (b < a) {
          a = b;
          ca = q;
        }
      }
      if (a >= x) break;
      put(p, a);
      p = ca;
    }
    put(p, x);
  }

  // Expand every lane's pending records into its heap, in two phases.
  // 1. Each lane lists, in key order, the elements of its own records that
  //    beat tau (one-byte codes: record slot * 8 + element); predicated
  //    stores, no cross-lane traffic.
  // 2. The warp walks the lists in lockstep, one element per lane per step,
  //    re-checking each against the current root: one heap replace body
  //    serves all lanes at once.
  __device__ __forceinline__ void flush() {
    int cnt = 0;
    for (int i = 0; i < rc; ++i) {
      const float4 a = rlo[i * ROWS];
      const float4 b = rhi[i * ROWS];
      const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        if (v[e] > tau) {
          stage[cnt * ROWS] = static_cast<uint8_t>(i * 8 + e);
          ++cnt;
        }
      }
    }
    const int mx = __reduce_max_sync(0xffffffffu, static_cast<unsigned>(cnt));
    // software-pipelined: the next element's loads are issued before this push
    auto fetch = [&](int t, float& x, uint32_t& j) {
      const int code = stage[t * ROWS];
      const int i = code >> 3, e = code & 7;
      x = reinterpret_cast<const float*>((e < 4 ? rlo : rhi) + i * ROWS)[e & 3];
      j = rj[i * ROWS] + static_cast<uint32_t>(e);
    };
    float x = -INFINITY;
    uint32_t j = 0;
    if (cnt > 0) fetch(0, x, j);
    for (int t = 0; t < mx; ++t) {
      float xn = -INFINITY;
      uint32_t jn = 0;
      if (t + 1 < cnt) fetch(t + 1, xn, jn);
      if (t < cnt && x > tau) push(make_key(x, j));
      x = xn;
      j = jn;
    }
    rc = 0;
  }

  // Offer W scores with key indices j0 .. j0+W-1 (ascending).  The maxima of
  // the W/8 groups are independent (computed first, for instruction-level
  // parallelism); each group that beats tau becomes one record; one warp
  // vote per call decides whether to flush, keeping every lane's record
  // count at most gr - W/8 between calls.
  template <int W>
  __device__ __forceinline__ void offer(const float (&v)[W], uint32_t j0) {
    constexpr int G = W / 8;
    float m[G];
#pragma unroll
    for (int g = 0; g < G; ++g)
      m[g] = max3f(max3f(v[8 * g], v[8 * g + 1], v[8 * g + 2]), max3f(v[8 * g + 3], v[8 * g + 4], v[8 * g + 5]),
                   fmaxf(v[8 * g + 6], v[8 * g + 7]));
    // branch-free: a group that does not beat tau is written to the scratch
    // slot gr (never read) and does not advance the count
    int r = rc;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const int pass = m[g] > tau ? 1 : 0;
      const int slot = pass ? r : gr;
      rlo[slot * ROWS] = make_float4(v[8 * g], v[8 * g + 1], v[8 * g + 2], v[8 * g + 3]);
      rhi[slot * ROWS] = make_float4(v[8 * g + 4], v[8 * g + 5], v[8 * g + 6], v[8 * g + 7]);
      rj[slot * ROWS] = j0 + 8 * g;
      r += pass;
    }
    rc = r;
    if (__any_sync(0xffffffffu, rc > gr - G)) flush();
  }

  // After the last key: merge what is pending, then heap-sort in place so
  // that slots 0 .. n-1 hold the kept keys in selection order (best first).
  // A row that never filled its heap (fewer than k valid keys) is heapified
  // first: its entries were appended unordered.
  __device__ __forceinline__ void finish() {
    flush();
    if constexpr (FIXED_K == 64) {
      if (n < k && n > 1)
        for (int p = (n - 2) / 8; p >= 0; --p) sift_down8(get(p), p, n);
      for (int m = n - 1; m > 0; --m) {
        const uint64_t x = get(m);
        put(m, get(0));
        sift_down8(x, 0, m);
      }
    } else {
      if (n < k && n > 1)
        for (int p = (n - 2) / 4; p >= 0; --p) sift_down(get(p), p, n);
      for (int m = n - 1; m > 0; --m) {
        const uint64_t x = get(m);
        put(m, get(0));
        sift_down(x, 0, m);
      }
    }
  }
};

// Replace scores of invalid keys (index >= lim) by -inf.
template <int W>
__device__ __forceinline__ void mask_scores(float (&v)[W], uint32_t j0, uint32_t lim) {
#pragma unroll
  for (int e = 0; e < W; ++e)
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
template <typename T, int D, typename Sel>
__device__ __forceinline__ void softmax_gather_store(const Sel& h, const T* __restrict__ vbase,
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
#pragma unroll 2
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
template <typename Sel>
__device__ __forceinline__ void write_selection(const Sel& h, int32_t* idx_row, float* score_row) {
  for (int t = 0; t < h.k; ++t) {
    const bool have = t < h.n;
    const uint64_t key = have ? h.get(t) : 0;
    if (idx_row) idx_row[t] = have ? static_cast<int32_t>(key_index(key)) : -1;
    if (score_row) score_row[t] = have ? key_score(key) : -INFINITY;
  }
}

}  // namespace topk
