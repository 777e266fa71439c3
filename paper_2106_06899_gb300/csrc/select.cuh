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

// The heap of one row: a min-heap of its k best packed keys in shared memory
// ([slot][row] layout, ROWS rows per slot).  push() offers one key; sort()
// turns the heap into the kept keys in selection order.  The 4-ary layout
// halves the dependent shared-memory round trips of a replace (log4 k levels
// of four independent loads).
template <int ROWS, int FIXED_K = 0>
struct HeapCore {
  // FIXED_K == 64: an 8-ary heap of exactly 64 keys, padded with 9 sentinel
  // slots (largest key) so that every interior node has 8 children: a root
  // replacement is two fully unrolled levels of 8 independent loads.
  // FIXED_K == 128: a two-level heap of any k in [65, 137] keys (k is a
  // runtime value): the root (slot 0), 8 nodes (slots 1..8) and up to 16
  // leaves under node c (slots 9 + 16 (c - 1) .. + 15 that are below k; a
  // missing leaf reads as the largest key).  A root replacement is 8 + 16
  // independent loads, without sentinel slots.
  static constexpr int kPad = FIXED_K == 64 ? 9 : 0;
  static constexpr int kLeaves = FIXED_K == 128 ? 16 : 8;  // children per level-1 node (fixed shapes)

  // slot of the q-th child of level-1 node c (1..8) in the fixed shapes
  __device__ __forceinline__ static int leaf_slot(int c, int q) {
    if constexpr (FIXED_K == 128)
      return 9 + 16 * (c - 1) + q;
    else
      return 8 * c + 1 + q;
  }
  // key at a leaf slot (the largest key where the two-level shape has none)
  __device__ __forceinline__ uint64_t leaf_key(int s) const {
    if constexpr (FIXED_K == 128)
      return s < k ? get(s) : ~0ull;
    else
      return get(s);
  }
  uint64_t* base;  // &heap[slot 0][this row]
  int k;           // capacity
  int n;           // entries filled
  uint64_t root;   // heap[0] once full
  float tau;       // score of heap[0] once full, else -inf

  __host__ __device__ static constexpr size_t heap_bytes(int k_) {
    return static_cast<size_t>(ROWS) * static_cast<size_t>(k_ + kPad) * 8;
  }

  __device__ __forceinline__ void init_heap(uint8_t* smem, int row, int cap) {
    base = reinterpret_cast<uint64_t*>(smem) + row;
    for (int q = 0; q < kPad; ++q) base[(cap + q) * ROWS] = ~0ull;  // sentinels never leave the leaves
    k = cap;
    n = 0;
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
  // hold sentinels.  Replace the root by x and restore the heap order;
  // returns the new root (the smaller of x and the root's smallest child),
  // so that the caller need not read it back.
  __device__ __forceinline__ uint64_t replace_root64(uint64_t x) {
    int p = 0;
    bool done = false;
    uint64_t new_root = x;
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
      if (level == 0 && a < x) new_root = a;
      if (!done && a < x) {
        put(p, a);
        p = ca;
      } else {
        done = true;
      }
    }
    put(p, x);
    return new_root;
  }

  // Branch-free form of replace_root64 for a full 8-ary heap of 64: if act,
  // x (which must rank above the root) replaces the root; both levels are
  // always read and the stores are predicated, so that a warp whose lanes
  // disagree on act runs one straight-line body.  Returns the root after
  // the call (`cur`, the current root, when act is false).
  __device__ __forceinline__ uint64_t replace_pred(uint64_t x, bool act, uint64_t cur) {
    uint64_t ch[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) ch[q] = get(1 + q);
    uint64_t a0;
    int i0;
    argmin8(ch, a0, i0);
    const int c0 = 1 + i0;
    const bool go0 = act && a0 < x;
    const int c1b = 8 * c0 + 1;
#pragma unroll
    for (int q = 0; q < 8; ++q) ch[q] = get(c1b + q);
    uint64_t a1;
    int i1;
    argmin8(ch, a1, i1);
    const bool go1 = go0 && a1 < x;
    const uint64_t top = go0 ? a0 : x;
    st_shared_u64_if(act, base, top);
    st_shared_u64_if(go0, base + c0 * ROWS, go1 ? a1 : x);
    st_shared_u64_if(go1, base + (c1b + i1) * ROWS, x);
    return act ? top : cur;
  }

  // replace_pred with the root (cur) and its 8 children (slots 1..8) kept
  // in registers by the caller across calls: level 0 needs no shared-memory
  // round trip, and only the leaf level is written to shared memory here.
  // The caller writes the root and ch0 back to slots 0..8 afterwards.
  __device__ __forceinline__ uint64_t replace_pred_rc(uint64_t x, bool act, uint64_t cur, uint64_t (&ch0)[8]) {
    uint64_t a0;
    int i0;
    argmin8(ch0, a0, i0);
    const int c0 = 1 + i0;
    const bool go0 = act && a0 < x;
    uint64_t ch[kLeaves];
#pragma unroll
    for (int q = 0; q < kLeaves; ++q) ch[q] = leaf_key(leaf_slot(c0, q));
    uint64_t a1;
    int i1;
    argmin_n(ch, a1, i1);
    const bool go1 = go0 && a1 < x;
    const uint64_t top = go0 ? a0 : x;
    const uint64_t mid = go1 ? a1 : x;
    st_shared_u64_if(go1, base + leaf_slot(c0, i1) * ROWS, x);
#pragma unroll
    for (int q = 0; q < 8; ++q) ch0[q] = (go0 && q == i0) ? mid : ch0[q];
    return act ? top : cur;
  }

  // Branch-free root replacement in a full 4-ary heap (FIXED_K == 0) of at
  // most 1364 keys: if act, x (which must rank above the root) replaces the
  // root.  Five levels are always walked with predicated stores, and a child
  // past k reads as the largest key, so lanes that disagree on act or on the
  // depth run one straight-line body.  Returns the root after the call (cur
  // when act is false).
  __device__ __forceinline__ uint64_t replace_pred4(uint64_t x, bool act, uint64_t cur) {
    int p = 0;
    bool go = act;
    uint64_t top = x;
#pragma unroll
    for (int level = 0; level < 5; ++level) {
      const int c = 4 * p + 1;
      uint64_t ch[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) ch[q] = c + q < k ? get(c + q) : ~0ull;
      const bool l01 = ch[0] <= ch[1], l23 = ch[2] <= ch[3];
      const uint64_t m01 = l01 ? ch[0] : ch[1], m23 = l23 ? ch[2] : ch[3];
      const int i01 = l01 ? 0 : 1, i23 = l23 ? 2 : 3;
      const bool lf = m01 <= m23;
      const uint64_t a = lf ? m01 : m23;
      const bool down = go && a < x;
      if (level == 0) top = down ? a : x;
      st_shared_u64_if(go, base + p * ROWS, down ? a : x);  // the child moves up, or x settles here
      p = down ? c + (lf ? i01 : i23) : p;
      go = down;
    }
    st_shared_u64_if(go, base + p * ROWS, x);  // below the fifth level
    return act ? top : cur;
  }

  // Smallest of NC keys (a power of two) and its first position (a tree).
  template <int NC>
  __device__ __forceinline__ static void argmin_n(const uint64_t (&ch)[NC], uint64_t& m, int& i) {
    uint64_t v[NC];
    int p[NC];
#pragma unroll
    for (int q = 0; q < NC; ++q) {
      v[q] = ch[q];
      p[q] = q;
    }
#pragma unroll
    for (int w = NC / 2; w >= 1; w /= 2) {
#pragma unroll
      for (int q = 0; q < w; ++q) {
        const bool lo = v[q] <= v[q + w];
        v[q] = lo ? v[q] : v[q + w];
        p[q] = lo ? p[q] : p[q + w];
      }
    }
    m = v[0];
    i = p[0];
  }

  // Sift x down from slot p in the two-level shape of k keys.
  __device__ __forceinline__ void sift128(uint64_t x, int p) {
    for (;;) {
      int first, cnt;
      if (p == 0) {
        first = 1;
        cnt = 8;
      } else if (p <= 8) {
        first = 9 + 16 * (p - 1);
        cnt = k - first < 16 ? k - first : 16;
        if (cnt <= 0) break;
      } else {
        break;
      }
      uint64_t a = get(first);
      int ca = first;
      for (int q = first + 1; q < first + cnt; ++q) {
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

  // Smallest of 8 keys and its position (tree of depth 3).
  __device__ __forceinline__ static void argmin8(const uint64_t (&ch)[8], uint64_t& m, int& i) {
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
    m = lf ? m01 : m23;
    i = lf ? i01 : i23;
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
        } else if constexpr (FIXED_K == 128) {
          for (int p = 8; p >= 0; --p) sift128(get(p), p);
        } else {
          for (int p = (k - 2) / 4; p >= 0; --p) sift_down(get(p), p, k);
        }
        root = get(0);
        tau = key_score(root);
      }
    } else if (x > root) {
      if constexpr (FIXED_K == 64) {
        root = replace_root64(x);
      } else if constexpr (FIXED_K == 128) {
        sift128(x, 0);
        root = get(0);
      } else {
        sift_down(x, 0, k);
        root = get(0);
      }
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

  // Heap-sort in place so that slots 0 .. n-1 hold the kept keys in
  // selection order (best first).  A row that never filled its heap (fewer
  // than k valid keys) is heapified first: its entries were appended
  // unordered.
  __device__ __forceinline__ void sort() {
    if constexpr (FIXED_K == 64) {
      if (n < k && n > 1)
        for (int p = (n - 2) / 8; p >= 0; --p) sift_down8(get(p), p, n);
      for (int m = n - 1; m > 0; --m) {
        const uint64_t x = get(m);
        put(m, get(0));
        sift_down8(x, 0, m);
      }
    } else {
      // the 4-ary order; the fixed 128 shape is not one, so it is rebuilt
      if ((n < k || FIXED_K == 128) && n > 1)
        for (int p = (n - 2) / 4; p >= 0; --p) sift_down(get(p), p, n);
      for (int m = n - 1; m > 0; --m) {
        const uint64_t x = get(m);
        put(m, get(0));
        sift_down(x, 0, m);
      }
    }
  }
};

// Exact per-row top-k for one warp that both filters and keeps the heap:
// HeapCore fed through a per-row buffer of pending score groups.
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
// re-checked at expansion.
// ROWS = number of rows sharing the [slot][row] arrays (the row stride);
// every call of offer*/flush/finish must be made by all 32 lanes of a warp.
template <int ROWS, int FIXED_K = 0>
struct RowHeap : HeapCore<ROWS, FIXED_K> {
  using Core = HeapCore<ROWS, FIXED_K>;
  using Core::kPad;
  using Core::push;
  using Core::tau;
  float4* rlo;     // &records_lo[0][this row]: scores 0..3
  float4* rhi;     // &records_hi[0][this row]: scores 4..7
  uint32_t* rj;    // &records_j0[0][this row]
  uint8_t* stage;  // &stage[0][this row]: codes (record slot * 8 + element) of elements to offer
  int rc;          // records pending
  int gr;          // record capacity

  // shared memory: heap (k + kPad) x ROWS x 8 bytes, records (gr + 1) x ROWS
  // x 36 bytes (the last one a scratch slot), stage 8 gr x ROWS bytes (gr <=
  // 31, so that a code fits in one byte)
  __host__ __device__ static constexpr size_t bytes(int k_, int gr_) {
    return Core::heap_bytes(k_) +
           static_cast<size_t>(ROWS) * (static_cast<size_t>(gr_ + 1) * 36 + static_cast<size_t>(gr_) * 8);
  }

  __device__ __forceinline__ void init(uint8_t* smem, int row, int cap, int rec_cap) {
    Core::init_heap(smem, row, cap);
    uint8_t* r = smem + Core::heap_bytes(cap);
    const size_t nrec = static_cast<size_t>(rec_cap) + 1;  // + scratch slot
    rlo = reinterpret_cast<float4*>(r) + row;
    rhi = reinterpret_cast<float4*>(r + nrec * ROWS * 16) + row;
    rj = reinterpret_cast<uint32_t*>(r + nrec * ROWS * 32) + row;
    stage = r + nrec * ROWS * 36 + row;
    gr = rec_cap;
    rc = 0;
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
    const bool fast = __all_sync(0xffffffffu, Core::n == Core::k);
    if constexpr (FIXED_K == 0) {
      if (fast) {  // every heap is full: one straight-line 4-ary replace per step
        uint64_t r = Core::root;
        for (int t = 0; t < mx; ++t) {
          float xn = -INFINITY;
          uint32_t jn = 0;
          if (t + 1 < cnt) fetch(t + 1, xn, jn);
          const uint64_t key = make_key(x, j);
          r = Core::replace_pred4(key, t < cnt && key > r, r);
          x = xn;
          j = jn;
        }
        Core::root = r;
        tau = key_score(r);
        rc = 0;
        return;
      }
    }
    if (FIXED_K != 0 && fast) {
      // every heap is full: one straight-line replace per step, the root and
      // its 8 children in registers, written back once
      uint64_t r = Core::root;
      uint64_t ch0[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) ch0[q] = Core::get(1 + q);
      for (int t = 0; t < mx; ++t) {
        float xn = -INFINITY;
        uint32_t jn = 0;
        if (t + 1 < cnt) fetch(t + 1, xn, jn);
        const uint64_t key = make_key(x, j);
        r = Core::replace_pred_rc(key, t < cnt && key > r, r, ch0);
        x = xn;
        j = jn;
      }
      Core::put(0, r);
#pragma unroll
      for (int q = 0; q < 8; ++q) Core::put(1 + q, ch0[q]);
      Core::root = r;
      tau = key_score(r);
    } else {
      for (int t = 0; t < mx; ++t) {
        float xn = -INFINITY;
        uint32_t jn = 0;
        if (t + 1 < cnt) fetch(t + 1, xn, jn);
        if (t < cnt && x > tau) push(make_key(x, j));
        x = xn;
        j = jn;
      }
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

  // After the last key: merge what is pending, then sort.
  __device__ __forceinline__ void finish() {
    flush();
    Core::sort();
  }
};

// ---------------------------------------------------------------------------
// Split selection: a filter warp and a heap warp share the same 32 rows.
//
// The filter warp reads the scores and keeps no heap: each group of 8 whose
// maximum beats its copy of the row's threshold goes, as one record (8 scores
// and the first key index), into the row's ring of R records.  The heap warp
// expands the records into the row's heap exactly as RowHeap::flush does and
// publishes the heap root's score as the new threshold.  Both warps run on
// the same SM sub-partition, so the heap work of one batch overlaps the
// filtering of the next instead of following it.
//
// Per row, in shared memory ([slot][row] like the heap):
//   end   u64  (unit sequence number << 32) | head at the unit's last record
//   tauw  u64  (unit sequence number << 32) | bits of the heap root's score
//   head  u32  records written (filter, release store)
//   tail  u32  records consumed (heap warp, release store)
//   R record slots, then kStage (score, index) pairs: the heap warp's own
//   list of the elements it is about to offer to the heap.  The heap warp
//   copies the qualifying elements out of the records first and frees the
//   slots at once, so that the filter refills the ring while the heap works.
// Counters are absolute and wrap modulo 2^32; the slot of record number c is
// c mod R (tracked incrementally).  Each unit (query tile) has a sequence
// number 1, 2, ... per CTA; a threshold or end mark of another unit is
// ignored.
template <int ROWS>
struct RingView {
  static constexpr int kStage = 16;
  uint64_t* end;
  uint64_t* tauw;
  uint32_t* head;
  uint32_t* tail;
  float4* lo;
  float4* hi;
  uint32_t* rj;
  uint2* stage;

  __host__ __device__ static constexpr size_t ctl_bytes() { return static_cast<size_t>(ROWS) * 24; }
  __host__ __device__ static constexpr size_t bytes(int R) {
    return ctl_bytes() + static_cast<size_t>(ROWS) * (static_cast<size_t>(R) * 36 + kStage * 8);
  }

  // mem must be 16-byte aligned; its first ctl_bytes() must be zero before use
  __device__ __forceinline__ void bind(uint8_t* mem, int row, int R) {
    end = reinterpret_cast<uint64_t*>(mem) + row;
    tauw = reinterpret_cast<uint64_t*>(mem + ROWS * 8) + row;
    head = reinterpret_cast<uint32_t*>(mem + ROWS * 16) + row;
    tail = reinterpret_cast<uint32_t*>(mem + ROWS * 20) + row;
    uint8_t* r = mem + ctl_bytes();
    const size_t nrec = static_cast<size_t>(R);
    lo = reinterpret_cast<float4*>(r) + row;
    hi = reinterpret_cast<float4*>(r + nrec * ROWS * 16) + row;
    stage = reinterpret_cast<uint2*>(r + nrec * ROWS * 32) + row;
    rj = reinterpret_cast<uint32_t*>(r + nrec * ROWS * 32 + kStage * ROWS * 8) + row;
  }
};

// Sleep between polls of a shared-memory counter: doubles from 32 ns to 512
// ns, so that a waiting warp leaves the issue slots of its SM sub-partition
// to the warp it waits for.
__device__ __forceinline__ unsigned backoff_ns(uint32_t polls) { return 32u << (polls < 4u ? polls : 4u); }

// Filter side.  Every call is made by all 32 lanes of the warp.
template <int ROWS>
struct RowFilter {
  RingView<ROWS> v;
  int R;
  uint32_t h;    // records written
  int hm;        // h mod R
  uint32_t tc;   // last tail seen
  uint32_t seq;  // current unit
  float tau;     // threshold: a lower bound of the row's final k-th score

  __device__ __forceinline__ void init(uint8_t* mem, int row, int R_) {
    v.bind(mem, row, R_);
    R = R_;
    h = 0;
    hm = 0;
    tc = 0;
    seq = 0;
  }

  __device__ __forceinline__ void begin_unit() {
    ++seq;
    tau = -INFINITY;
  }

  // Adopt the heap warp's threshold if it belongs to this unit.
  __device__ __forceinline__ void refresh_tau() {
    const uint64_t w = ld_relaxed_u64(v.tauw);
    if (static_cast<uint32_t>(w >> 32) == seq) tau = fmaxf(tau, __uint_as_float(static_cast<uint32_t>(w)));
  }

  // Waits (bounded) until every lane has room for `need` more records.
  // Everything written so far is published first: the heap warp may be
  // waiting for a fuller batch than it can see.
  __device__ __forceinline__ bool reserve(int need, const DevCtl& ctl, volatile int* abort_flag) {
    if (__all_sync(0xffffffffu, static_cast<int>(h - tc) + need <= R)) return true;
    publish();
    unsigned long long t0 = 0;
    for (uint32_t spin = 0;; ++spin) {
      tc = ld_acquire_u32(v.tail);
      if (__all_sync(0xffffffffu, static_cast<int>(h - tc) + need <= R)) return true;
      int stop = 0;
      if ((threadIdx.x & 31) == 0 && (spin & 15u) == 0) {
        if (spin == 0) {
          t0 = global_ns();
        } else if (*abort_flag) {
          stop = 1;
        } else if (global_ns() - t0 > ctl.wait_limit_ns) {
          atomicOr(ctl.error, kDevErrTimeout);
          *abort_flag = 1;
          stop = 1;
        }
      }
      if (__shfl_sync(0xffffffffu, stop, 0)) return false;
      __nanosleep(backoff_ns(spin));
    }
  }

  // Offer W scores with key indices j0 .. j0+W-1; needs W/8 free slots.
  // A group that does not pass costs no shared-memory store.
  template <int W>
  __device__ __forceinline__ void offer(const float (&x)[W], uint32_t j0) {
    constexpr int G = W / 8;
    float m[G];
#pragma unroll
    for (int g = 0; g < G; ++g)
      m[g] = max3f(max3f(x[8 * g], x[8 * g + 1], x[8 * g + 2]), max3f(x[8 * g + 3], x[8 * g + 4], x[8 * g + 5]),
                   fmaxf(x[8 * g + 6], x[8 * g + 7]));
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const bool pass = m[g] > tau;
      if (pass) {  // compiled to predicated stores
        v.lo[hm * ROWS] = make_float4(x[8 * g], x[8 * g + 1], x[8 * g + 2], x[8 * g + 3]);
        v.hi[hm * ROWS] = make_float4(x[8 * g + 4], x[8 * g + 5], x[8 * g + 6], x[8 * g + 7]);
        v.rj[hm * ROWS] = j0 + 8 * g;
      }
      const int nx = hm + (pass ? 1 : 0);
      hm = nx == R ? 0 : nx;
      h += pass ? 1u : 0u;
    }
  }

  // Make the records written so far visible to the heap warp.
  __device__ __forceinline__ void publish() { st_release_u32(v.head, h); }

  // Mark the end of this unit's records.  The heap warp must have taken the
  // previous unit's end mark first (it says so by publishing a threshold word
  // of this unit when it starts it): the end word has one slot.
  __device__ __forceinline__ bool end_unit(const DevCtl& ctl, volatile int* abort_flag) {
    unsigned long long t0 = 0;
    for (uint32_t spin = 0;; ++spin) {
      const uint32_t s = static_cast<uint32_t>(ld_acquire_u64(v.tauw) >> 32);
      if (__all_sync(0xffffffffu, s == seq)) break;
      int stop = 0;
      if ((threadIdx.x & 31) == 0 && (spin & 15u) == 0) {
        if (spin == 0) {
          t0 = global_ns();
        } else if (*abort_flag) {
          stop = 1;
        } else if (global_ns() - t0 > ctl.wait_limit_ns) {
          atomicOr(ctl.error, kDevErrTimeout);
          *abort_flag = 1;
          stop = 1;
        }
      }
      if (__shfl_sync(0xffffffffu, stop, 0)) return false;
      __nanosleep(backoff_ns(spin));
    }
    st_release_u64(v.end, (static_cast<uint64_t>(seq) << 32) | h);
    return true;
  }
};

// Heap side: HeapCore fed from the ring.  Every call is made by all 32 lanes.
template <int ROWS, int FIXED_K = 0>
struct RowSink : HeapCore<ROWS, FIXED_K> {
  using Core = HeapCore<ROWS, FIXED_K>;
  using Core::push;
  using Core::tau;
  using Core::n;
  using Core::k;
  RingView<ROWS> v;
  int R;
  uint32_t t;    // records consumed
  int tm;        // t mod R
  uint32_t seq;  // current unit

  __device__ __forceinline__ void init(uint8_t* ring_mem, int row, int R_) {
    v.bind(ring_mem, row, R_);
    R = R_;
    t = 0;
    tm = 0;
    seq = 0;
  }

  // Start the next unit: empty heap, and a threshold word of the new unit
  // (-inf), which also tells the filter warp that the previous end mark has
  // been taken.
  __device__ __forceinline__ void begin_unit(uint8_t* heap_mem, int row, int cap) {
    ++seq;
    Core::init_heap(heap_mem, row, cap);
    st_release_u64(v.tauw, (static_cast<uint64_t>(seq) << 32) | __float_as_uint(-INFINITY));
  }

  // Expand records t .. lim-1 into the heap, in two phases.
  // 1. Each lane copies the elements of its records that beat tau into its
  //    stage (predicated stores, in key order), as many records as the stage
  //    surely holds, then frees those ring slots.
  // 2. The warp walks the stages in lockstep, one element per lane per step,
  //    re-checking each against the current root.
  // Then the new threshold is published.
  __device__ __forceinline__ void consume(uint32_t lim) {
    constexpr int SC = RingView<ROWS>::kStage;
    const float thr = tau;  // -inf while the heap is filling
    int cnt = 0;
    int s = tm;
    uint32_t tt = t;
    while (tt != lim && cnt + 8 <= SC) {
      const float4 a = v.lo[s * ROWS];
      const float4 b = v.hi[s * ROWS];
      const uint32_t j0 = v.rj[s * ROWS];
      const float e8[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const bool pass = e8[e] > thr;
        st_shared_u2_if(pass, v.stage + cnt * ROWS, __float_as_uint(e8[e]), j0 + e);
        cnt += pass ? 1 : 0;
      }
      s = s + 1 == R ? 0 : s + 1;
      ++tt;
    }
    tm = s;
    t = tt;
    st_release_u32(v.tail, t);
    const int mx = __reduce_max_sync(0xffffffffu, static_cast<unsigned>(cnt));
    uint2 c = cnt > 0 ? v.stage[0] : make_uint2(0u, 0u);
    const bool fast = __all_sync(0xffffffffu, n == k);
    if (FIXED_K == 0 && fast) {  // every kept set is full: one straight-line 4-ary replace per step
      uint64_t r = Core::root;
      for (int q = 0; q < mx; ++q) {
        const uint2 cn = q + 1 < cnt ? v.stage[(q + 1) * ROWS] : make_uint2(0u, 0u);
        const uint64_t key = make_key(__uint_as_float(c.x), c.y);
        r = Core::replace_pred4(key, q < cnt && key > r, r);
        c = cn;
      }
      Core::root = r;
      tau = key_score(r);
    } else if (FIXED_K != 0 && fast) {
      // every kept set is full: one straight-line replace per step
      uint64_t r = Core::root;
      uint64_t ch0[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) ch0[q] = Core::get(1 + q);
      for (int q = 0; q < mx; ++q) {
        const uint2 cn = q + 1 < cnt ? v.stage[(q + 1) * ROWS] : make_uint2(0u, 0u);
        const uint64_t key = make_key(__uint_as_float(c.x), c.y);
        r = Core::replace_pred_rc(key, q < cnt && key > r, r, ch0);
        c = cn;
      }
      Core::put(0, r);
#pragma unroll
      for (int q = 0; q < 8; ++q) Core::put(1 + q, ch0[q]);
      Core::root = r;
      tau = key_score(r);
    } else {
      for (int q = 0; q < mx; ++q) {
        const uint2 cn = q + 1 < cnt ? v.stage[(q + 1) * ROWS] : make_uint2(0u, 0u);
        const float x = __uint_as_float(c.x);
        if (q < cnt && x > tau) push(make_key(x, c.y));
        c = cn;
      }
    }
    if (n == k) st_relaxed_u64(v.tauw, (static_cast<uint64_t>(seq) << 32) | __float_as_uint(tau));
  }

  // Consume this unit's records until its end mark has been seen and every
  // record before it expanded.  A batch starts when some row has `batch`
  // records pending (larger batches keep more lanes busy in the lockstep
  // expansion) or when the unit's records are all in.  `batch` must not
  // exceed the free-slot margin the filter waits for, or both would wait.
  // Returns false if the CTA aborts or nothing happens within the wait limit.
  __device__ __forceinline__ bool drain_unit(int batch, const DevCtl& ctl, volatile int* abort_flag) {
    unsigned long long t0 = 0;
    uint32_t idle = 0;
    for (;;) {
      // head before end: a head that already counts records of the next
      // unit implies that this unit's end mark is visible
      const uint32_t hd = ld_acquire_u32(v.head);
      const uint64_t e = ld_acquire_u64(v.end);
      const bool fin = static_cast<uint32_t>(e >> 32) == seq;
      const uint32_t lim = fin ? static_cast<uint32_t>(e) : hd;
      const int pend = static_cast<int>(lim - t);
      const bool all_fin = __all_sync(0xffffffffu, fin);
      if (__any_sync(0xffffffffu, pend >= batch) || (all_fin && __any_sync(0xffffffffu, pend != 0))) {
        consume(lim);
        idle = 0;
        continue;
      }
      if (all_fin) return true;
      int stop = 0;
      if ((threadIdx.x & 31) == 0 && (idle & 15u) == 0) {
        if (idle == 0) {
          t0 = global_ns();
        } else if (*abort_flag) {
          stop = 1;
        } else if (global_ns() - t0 > ctl.wait_limit_ns) {
          atomicOr(ctl.error, kDevErrTimeout);
          *abort_flag = 1;
          stop = 1;
        }
      }
      if (__shfl_sync(0xffffffffu, stop, 0)) return false;
      __nanosleep(backoff_ns(idle));
      ++idle;
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
// for one row, in any order of its kept entries.  Values are rows of D elements of
// type T (float or bf16) starting at `vbase` (row j at vbase + j * D); the
// result is written to `orow` (D elements of T).  Accumulation is fp32 over
// 64-column slices so that at most 64 accumulators are live.
template <typename T, int D, typename Sel>
__device__ __forceinline__ void softmax_gather_store(const Sel& h, const T* __restrict__ vbase,
                                                     T* __restrict__ orow) {
  constexpr int SL = D < 64 ? D : 64;
  const int n = h.n;
  float m = -INFINITY;  // the largest kept score, for a stable exponent
  for (int t = 0; t < n; ++t) m = fmaxf(m, key_score(h.get(t)));
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
