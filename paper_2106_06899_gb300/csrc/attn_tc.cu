// attn_tc.cu -- fused top-k attention (Eq. 4) for bf16 inputs on sm_103a.
//
// One persistent CTA per SM walks work units (b, h, 128-query tile).  For a
// unit the query tile Q_C (Sec. 2.2 "Query chunking", C = 128) is loaded once
// by TMA, then the keys stream through in tiles of N:
//
//   warp 0      TMA producer: Q tile, then K tiles into a shared-memory ring
//   warp 1      MMA issuer: S = Q_C K_tile^T with tcgen05.mma (bf16 in, fp32
//               accumulate) into one of two TMEM accumulators [128 x N]
//   warps 2..5  selection: thread t of warp w owns TMEM lane / query row
//               32*(w%4)+t; it reads its N scores with tcgen05.ld and offers
//               them to its row's top-k heap (select.cuh); after the last
//               key tile it sorts the k kept keys, applies the softmax over
//               them and gathers the matching value rows (fp32 accumulate).
//
// Split variant (when the heaps and a record ring fit in shared memory):
//   warps 2..5  filter: read the scores from TMEM and pass the groups of 8
//               that beat the row's threshold into the row's record ring
//   warps 6..9  heap: warp w serves the rows of warp w-4 (same TMEM lane
//               quarter, same SM sub-partition); it expands the records into
//               the heaps and publishes the rising threshold.  After the
//               unit's last record it parks the kept keys in a small device
//               buffer (two slots per warp) and starts the next unit at once,
//               when its filter warp sends the most records.
//   warps 10,11 epilogue: warp 10 + e takes the parked keys of the rows of
//               lane quarters 2e and 2e+1, applies the softmax over them and
//               gathers the matching value rows.
//
// The score tile never leaves TMEM/registers: no [C x Lk] matrix is written
// to device memory (Sec. 2.2 "Query chunking": memory O(C Lk) becomes
// O(C k) here, in shared memory).  The scale of Eq. 1 is folded into Q by
// the caller.  Causal masking (Eq. 2) skips key tiles past the query tile
// and masks keys j > i inside the diagonal tile.
//
// Every pipeline wait is bounded (common.cuh); on expiry the CTA stops,
// drains its in-flight copies and MMAs, frees TMEM and returns.
#include <algorithm>

#include "kernels.h"
#include "select.cuh"

namespace topk {

namespace {

constexpr int BM = 128;
template <bool SPLIT>
constexpr int kThreads = SPLIT ? 384 : 192;  // split: 12 warps, three per SM sub-partition

// Parked kept keys of the split kernel, per CTA: 4 heap warps x 2 slots x
// topk keys x 32 rows (8 bytes each), then the kept count of each row.
__host__ __device__ constexpr size_t park_keys_per_cta(int topk) { return static_cast<size_t>(4) * 2 * topk * 32; }
__host__ __device__ constexpr size_t park_bytes(int grid, int topk) {
  return static_cast<size_t>(grid) * (park_keys_per_cta(topk) * 8 + 4 * 2 * 32 * 4);
}

template <int D, bool SPLIT>
struct TcShape;
// N: keys per tile (MMA N); S: key-ring stages; OW: scores per selection call.
// The split variant takes smaller key tiles to leave room for its record ring.
template <bool SPLIT>
struct TcShape<64, SPLIT> {
  static constexpr int N = SPLIT ? 128 : 256;
  static constexpr int S = 2;
  static constexpr int OW = 32;
};
template <bool SPLIT>
struct TcShape<128, SPLIT> {
  static constexpr int N = 64;
  static constexpr int S = 2;
  // One group of 8 per selection call: with a 128-key heap per row (128 KB),
  // a 32 KB Q tile and two 16 KB key stages, a row's ring (or record buffer)
  // gets only a few slots, and a call that needs fewer of them stalls and
  // flushes less often (causal_16k: 21.8 ms with 32 scores per call, 16.0 ms
  // with 8).
  static constexpr int OW = 8;
};

// RPU: query rows per work unit.  The MMA tile always has BM = 128 rows; with
// RPU = 64 or 32 (single-warp kernel only) just the first RPU of them belong
// to the unit, so that one row's heap can hold 256 or 512 keys: the heaps of
// RPU rows of k keys take RPU * k * 8 bytes of shared memory.
template <int D, int FK, bool SPLIT, int RPU = BM>
struct Layout {
  static_assert(RPU == BM || !SPLIT, "reduced-row units run the single-warp kernel");
  using Sel = RowHeap<RPU, FK>;
  using Heap = HeapCore<RPU, FK>;
  using Ring = RingView<BM>;
  static constexpr int N = TcShape<D, SPLIT>::N;
  static constexpr int S = TcShape<D, SPLIT>::S;
  // the two-level heap of 65 <= k <= 137 (up to 137 KB) leaves a row only a
  // few ring or record slots: one group of 8 per selection call, so that a
  // call needs one slot (see TcShape<128>)
  static constexpr int OW = FK == 128 ? 8 : TcShape<D, SPLIT>::OW;
  static constexpr int R = D / 64;  // 128-byte column blocks per row
  static constexpr uint32_t Q_BYTES = BM * D * 2;
  static constexpr uint32_t KST_BYTES = N * D * 2;
  static constexpr size_t OFF_Q = 0;
  static constexpr size_t OFF_K = OFF_Q + Q_BYTES;
  static constexpr size_t OFF_SEL = OFF_K + static_cast<size_t>(S) * KST_BYTES;
  // TMEM accumulators: as many N-column buffers as fit in 512 columns, at
  // most 4, so that the MMA warp can run ahead of a selection that stalls
  static constexpr int NACC = 512 / N < 4 ? 512 / N : 4;
  static constexpr int NBARS = 2 * S + 3 + 2 * NACC;
  static constexpr size_t CTRL_BYTES = 256;
  static constexpr size_t kMaxSmem = 232448;
  static constexpr size_t kFixed = 1024 + OFF_SEL + CTRL_BYTES;

  // Single-warp selection: pending score groups per row, as many as fit, at
  // most 24; a selection call adds up to OW/8 groups, so fewer than OW/8 + 1
  // does not work (0).  Split selection: record ring slots per row, at most
  // 24; the filter reserves OW/8 slots per selection call and the heap warp
  // starts a batch at 2R/3 pending (rounded down), which must not exceed
  // R - OW/8 + 1 (else both could wait): R >= 3 (OW/8 - 1); at least 2 OW/8.
  static constexpr int kMinCap = SPLIT ? 2 * (OW / 8) : OW / 8 + 1;
  static_assert(!SPLIT || 2 * kMinCap / 3 <= kMinCap - OW / 8 + 1, "batch threshold above the filter margin");
  __host__ __device__ static constexpr size_t heap_bytes(int topk) {
    return (Heap::heap_bytes(topk) + 15) & ~size_t(15);
  }
  __host__ __device__ static size_t sel_bytes(int topk, int cap) {
    if constexpr (SPLIT)
      return heap_bytes(topk) + ((Ring::bytes(cap) + 15) & ~size_t(15));
    else
      return (Sel::bytes(topk, cap) + 15) & ~size_t(15);
  }
  static int cap(int topk) {
    if (kFixed + sel_bytes(topk, kMinCap) > kMaxSmem) return 0;
    int c = kMinCap;
    while (c < 24 && kFixed + sel_bytes(topk, c + 1) <= kMaxSmem) ++c;
    return c;
  }
  static bool fits(int topk) { return cap(topk) >= kMinCap; }
  static size_t bytes(int topk) { return kFixed + sel_bytes(topk, cap(topk)); }
};

// Waits on an mbarrier phase with lane 0 of the warp and broadcasts the
// outcome, so that the whole warp leaves together.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, const DevCtl& ctl,
                                          volatile int* abort_flag) {
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ctl, abort_flag) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  return ok != 0;
}

// Waits (bounded; lane 0 polls) until the shared-memory counter *ctr, which
// only grows, reaches target; every lane then reads it with acquire
// semantics itself, so that what the releasing warp wrote before it is
// visible to the whole warp.  False if the CTA aborts or the limit runs out.
__device__ __forceinline__ bool wait_count(uint32_t* ctr, uint32_t target, const DevCtl& ctl,
                                           volatile int* abort_flag) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0 && static_cast<int>(ld_acquire_u32(ctr) - target) < 0) {
    const unsigned long long t0 = global_ns();
    for (uint32_t spin = 0;; ++spin) {
      if (static_cast<int>(ld_acquire_u32(ctr) - target) >= 0) break;
      if ((spin & 15u) == 15u) {
        if (*abort_flag) {
          ok = 0;
          break;
        }
        if (global_ns() - t0 > ctl.wait_limit_ns) {
          atomicOr(ctl.error, kDevErrTimeout);
          *abort_flag = 1;
          ok = 0;
          break;
        }
      }
      __nanosleep(backoff_ns(spin));
    }
  }
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (ok) (void)ld_acquire_u32(ctr);
  return ok != 0;
}

// The kept keys of one row as parked by its heap warp (every 32nd word),
// read through L2: they were written by another warp of the CTA.
struct ParkedKeys {
  const uint64_t* p;
  int n;
  __device__ __forceinline__ uint64_t get(int t) const {
    return __ldcg(reinterpret_cast<const unsigned long long*>(p) + static_cast<size_t>(t) * 32);
  }
};

// Bounded wait that ignores the abort flag: used only to drain in-flight
// asynchronous work before the CTA exits.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity, const DevCtl& ctl) {
  const unsigned long long t0 = global_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_ns() - t0 > ctl.wait_limit_ns) {
      atomicOr(ctl.error, kDevErrTimeout);
      return;
    }
  }
}

template <int D, int FK, bool SPLIT, int RPU = BM>
__global__ void __launch_bounds__(kThreads<SPLIT>, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmk,
                   const __nv_bfloat16* __restrict__ v, __nv_bfloat16* __restrict__ out, int BH, int H, int Lq,
                   int Lk, int topk, int rec_cap, int causal, const int32_t* __restrict__ kv_len, int n_units,
                   int parts, uint64_t* __restrict__ part_keys, int* __restrict__ part_n, int32_t* __restrict__ idx,
                   float* __restrict__ score, uint64_t* __restrict__ park, int* __restrict__ park_n, DevCtl ctl) {
  using L = Layout<D, FK, SPLIT, RPU>;
  using Sel = typename L::Sel;
  constexpr int N = L::N, S = L::S, R = L::R;
  constexpr uint32_t IDESC = idesc_bf16_f32(BM, N);
  constexpr int NACC = L::NACC;
  constexpr uint32_t TMEM_COLS = NACC * N;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* q_s = smem + L::OFF_Q;
  uint8_t* k_s = smem + L::OFF_K;
  uint8_t* sel_mem = smem + L::OFF_SEL;
  uint8_t* ring_mem = sel_mem + L::heap_bytes(topk);  // split variant only
  uint64_t* bars = reinterpret_cast<uint64_t*>(sel_mem + L::sel_bytes(topk, rec_cap));
  uint64_t* full_k = bars;
  uint64_t* empty_k = bars + S;
  uint64_t* q_full = bars + 2 * S;
  uint64_t* q_empty = bars + 2 * S + 1;
  uint64_t* acc_full = bars + 2 * S + 2;          // [NACC]
  uint64_t* acc_empty = bars + 2 * S + 2 + NACC;  // [NACC]
  uint64_t* drain = bars + 2 * S + 2 + 2 * NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + L::NBARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* pk_done = tmem_slot + 2;  // [4] split: units parked by each heap warp
  uint32_t* ep_done = tmem_slot + 6;  // [4] split: units finished by the epilogue, per lane quarter

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_k[s], 1);
      mbar_init(&empty_k[s], 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int b = 0; b < NACC; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    for (int q = 0; q < 4; ++q) pk_done[q] = ep_done[q] = 0;
    fence_mbar_init();
  }
  if constexpr (SPLIT) {  // ring counters, end marks and thresholds start at 0
    uint32_t* z = reinterpret_cast<uint32_t*>(ring_mem);
    for (int i = threadIdx.x; i < static_cast<int>(L::Ring::ctl_bytes() / 4); i += blockDim.x) z[i] = 0;
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_qt = (Lq + RPU - 1) / RPU;
  // A unit is (b, h, query tile, key part): with parts > 1 (grids that would
  // leave SMs idle, as decoding a few positions against a long cache does)
  // each query tile's key tiles are split into `parts` ranges, each part keeps
  // its own top k, and a merge kernel combines them.
  auto decode = [&](int u_, int& bh, int& qt, int& part) {
    part = u_ % parts;
    const int u = u_ / parts;
    if (causal) {  // heaviest query tiles first
      qt = n_qt - 1 - u / BH;
      bh = u % BH;
    } else {  // consecutive units share a head, so its K/V stay in L2
      bh = u / n_qt;
      qt = u % n_qt;
    }
  };
  // Eq. 2's masks as a valid key prefix per row: causal (queries are the
  // last Lq positions: key j is valid for query i iff j <= i + Lk - Lq) and
  // the batch's key count.  A unit streams at least one key tile, all of it
  // masked if its rows have no key, so that every pipeline stage runs.
  const int coff = Lk - Lq;
  auto kv_end = [&](int bh) { return kv_len ? min(max(__ldg(kv_len + bh / H), 0), Lk) : Lk; };
  auto key_tiles = [&](int bh, int qt) {
    int kend = min(kv_end(bh), causal ? (qt + 1) * RPU + coff : Lk);
    kend = max(kend, 1);
    return (kend + N - 1) / N;
  };
  auto row_limit = [&](int bh, int i) {  // keys j < limit are valid for query i
    return static_cast<uint32_t>(min(kv_end(bh), causal ? min(i + 1 + coff, Lk) : Lk));
  };
  auto tile_limit_min = [&](int bh, int qt) {  // the smallest row limit of query tile qt
    return min(kv_end(bh), causal ? min(qt * RPU + 1 + coff, Lk) : Lk);
  };
  // key tiles [t0, t1) of a unit's part; a part left without tiles streams one
  // fully masked tile (empty = true) so that every stage keeps its handshakes
  auto tile_range = [&](int bh, int qt, int part, int& t0, int& t1, bool& empty) {
    const int nk = key_tiles(bh, qt);
    t0 = static_cast<int>(static_cast<long long>(part) * nk / parts);
    t1 = static_cast<int>(static_cast<long long>(part + 1) * nk / parts);
    empty = t1 <= t0;
    if (empty) {
      t0 = 0;
      t1 = 1;
    }
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmq);
      tma_prefetch_desc(&tmk);
    }
    uint32_t it = 0, q_issued = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      if (!warp_wait(q_empty, (q_issued & 1u) ^ 1u, ctl, abort_flag)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(q_full, L::Q_BYTES);
        for (int r = 0; r < R; ++r) tma_load_3d(q_s + r * BM * 128, &tmq, q_full, r * 64, qt * RPU, bh);
      }
      ++q_issued;
      int t0, t1;
      bool empty;
      tile_range(bh, qt, part, t0, t1, empty);
      for (int kt = t0; kt < t1; ++kt) {
        const int s = it % S;
        const uint32_t ph = (it / S) & 1u;
        if (!warp_wait(&empty_k[s], ph ^ 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          if (ctl.debug_skip_arrive && it == 1) {
            // testing hook: withhold this stage so the consumers' waits run out
          } else {
            mbar_arrive_expect_tx(&full_k[s], L::KST_BYTES);
            for (int r = 0; r < R; ++r)
              tma_load_3d(k_s + static_cast<size_t>(s) * L::KST_BYTES + r * N * 128, &tmk, &full_k[s], r * 64,
                          kt * N, bh);
          }
        }
        ++it;
      }
    }
    // drain: every issued copy must have landed before the CTA may exit
    if (lane == 0) {
      for (uint32_t back = 1; back <= static_cast<uint32_t>(S) && back <= it; ++back) {
        const uint32_t t = it - back;
        if (ctl.debug_skip_arrive && t == 1) continue;
        mbar_drain(&full_k[t % S], (t / S) & 1u, ctl);
      }
      if (q_issued > 0) mbar_drain(q_full, (q_issued - 1) & 1u, ctl);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    uint32_t it = 0, acc_it = 0, qi = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x, ++qi) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      if (!warp_wait(q_full, qi & 1u, ctl, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      int t0, t1;
      bool empty;
      tile_range(bh, qt, part, t0, t1, empty);
      for (int kt = t0; kt < t1; ++kt, ++it, ++acc_it) {
        const int s = it % S;
        if (!warp_wait(&full_k[s], (it / S) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        const int b = acc_it % NACC;
        if (!warp_wait(&acc_empty[b], ((acc_it / NACC) & 1u) ^ 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (lane == 0) {
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(b * N);
          const uint32_t qa = smem_u32(q_s);
          const uint32_t ka = smem_u32(k_s + static_cast<size_t>(s) * L::KST_BYTES);
#pragma unroll
          for (int st = 0; st < D / 16; ++st) {
            const uint32_t r = st / 4, off = (st % 4) * 32;
            mma_bf16_ss(d_tmem, sdesc_k128(qa + r * BM * 128 + off), sdesc_k128(ka + r * N * 128 + off), IDESC,
                        st > 0 ? 1u : 0u);
          }
          mma_commit(&empty_k[s]);
          mma_commit(&acc_full[b]);
        }
        __syncwarp();
      }
      if (!ok) break;
      if (lane == 0) mma_commit(q_empty);
      __syncwarp();
    }
    // drain: all issued MMAs must complete before TMEM is freed
    if (lane == 0) {
      mma_commit(drain);
      mbar_drain(drain, 0, ctl);
    }
    __syncwarp();
  } else if (SPLIT && warp < 6) {
    // ------------------------------------------------------------ filter (split)
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    constexpr int OW = L::OW;
    uint32_t acc_it = 0;
    RowFilter<BM> f;
    f.init(ring_mem, row, rec_cap);
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      f.begin_unit();
      const int i_row = qt * BM + row;
      int t0, t1;
      bool empty;
      tile_range(bh, qt, part, t0, t1, empty);
      const uint32_t lim = empty ? 0u : row_limit(bh, i_row);
      const int lim_min = empty ? 0 : tile_limit_min(bh, qt);
      for (int kt = t0; ok && kt < t1; ++kt, ++acc_it) {
        const int b = acc_it % NACC;
        if (!warp_wait(&acc_full[b], (acc_it / NACC) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(b * N);
        const uint32_t jt = static_cast<uint32_t>(kt * N);
        f.refresh_tau();
        if constexpr (N == 128) {
          // both 64-column halves into separate registers up front: the
          // second load never waits for the first half's record stores
          float va[64], vb[64];
          __syncwarp();
          tmem_ld64(taddr, va);
          tmem_ld64(taddr + 64, vb);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);
          if (static_cast<int>(jt) + 64 > lim_min) mask_scores(va, jt, lim);
          if (static_cast<int>(jt) + 128 > lim_min) mask_scores(vb, jt + 64u, lim);
          constexpr int HALF = 64 / OW;  // calls per 64-column half
#pragma unroll
          for (int h = 0; h < 2 * HALF && ok; ++h) {
            if (!f.reserve(OW / 8, ctl, abort_flag)) {
              ok = false;
              break;
            }
            const float* src = h < HALF ? va + h * OW : vb + (h - HALF) * OW;
            f.offer(*reinterpret_cast<const float(*)[OW]>(src), jt + static_cast<uint32_t>(h * OW));
          }
        } else {
#pragma unroll 1
          for (int c = 0; c < N / 64 && ok; ++c) {
            float vals[64];
            __syncwarp();
            tmem_ld64(taddr + c * 64, vals);
            tmem_wait_ld();
            if (c == N / 64 - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);
            }
            const uint32_t j0 = jt + static_cast<uint32_t>(c * 64);
            if (static_cast<int>(j0) + 64 > lim_min) mask_scores(vals, j0, lim);
#pragma unroll
            for (int h = 0; h < 64 / OW; ++h) {
              if (!f.reserve(OW / 8, ctl, abort_flag)) {
                ok = false;
                break;
              }
              f.offer(reinterpret_cast<const float(&)[OW]>(vals[h * OW]), j0 + static_cast<uint32_t>(h * OW));
            }
          }
        }
        if (!ok) break;
        f.publish();  // once per key tile
      }
      if (ok && !f.end_unit(ctl, abort_flag)) ok = false;
    }
  } else if (SPLIT && warp < 10) {
    // ------------------------------------------------------------ heap (split)
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    RowSink<BM, FK> heap;
    heap.init(ring_mem, row, rec_cap);
    const size_t park0 = (static_cast<size_t>(blockIdx.x) * 4 + quad) * 2;  // this warp's first slot
    uint32_t s = 0;                                                           // units done by this warp
    for (int u = blockIdx.x; u < n_units; u += gridDim.x, ++s) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      const int i_row = qt * BM + row;
      heap.begin_unit(sel_mem, row, topk);
      // batch threshold: two thirds of the ring, within the filter's margin
      // of OW/8 free slots, so that the filter never waits on a heap warp
      // that waits
      if (!heap.drain_unit(rec_cap * 2 / 3, ctl, abort_flag)) break;
      if (i_row < Lq && (idx || score)) {  // only the index/score outputs need the order
        const size_t orow = static_cast<size_t>(bh) * Lq + i_row;
        heap.sort();
        write_selection(heap, idx ? idx + orow * topk : nullptr, score ? score + orow * topk : nullptr);
      }
      // park the kept keys in slot s % 2; it last held unit s - 2, whose
      // epilogue must be done
      if (s >= 2 && !wait_count(&ep_done[quad], s - 1, ctl, abort_flag)) break;
      const size_t slot = park0 + (s & 1u);
      uint64_t* pk = park + slot * topk * 32 + lane;
      const int n = i_row < Lq ? heap.n : 0;
      for (int t = 0; t < n; ++t) pk[static_cast<size_t>(t) * 32] = heap.get(t);
      park_n[slot * 32 + lane] = n;
      __syncwarp();
      st_release_u32(&pk_done[quad], s + 1);
    }
  } else if (SPLIT) {
    // ------------------------------------------------------------ epilogue (split)
    // Warp 10 + e finishes the rows of lane quarters 2e and 2e + 1, unit by
    // unit: the softmax over each row's parked kept keys (any order) and the
    // weighted sum of their value rows.
    const int e = warp - 10;
    uint32_t s = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x, ++s) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      for (int h = 0; h < 2; ++h) {
        const int q = 2 * e + h;
        if (!wait_count(&pk_done[q], s + 1, ctl, abort_flag)) {
          ok = false;
          break;
        }
        const int i_row = qt * BM + q * 32 + lane;
        const size_t slot = (static_cast<size_t>(blockIdx.x) * 4 + q) * 2 + (s & 1u);
        const int n = __ldcg(park_n + slot * 32 + lane);
        if (i_row < Lq) {  // a row without a valid key (n = 0) gets zeros
          const size_t orow = static_cast<size_t>(bh) * Lq + i_row;
          const ParkedKeys kept{park + slot * topk * 32 + lane, n};
          if (parts > 1) {  // this part's kept keys, for the merge
            const size_t prow = static_cast<size_t>(part) * BH * Lq + orow;
            for (int t = 0; t < n; ++t) part_keys[prow * topk + t] = kept.get(t);
            part_n[prow] = n;
          } else {
            softmax_gather_store<__nv_bfloat16, D>(kept, v + static_cast<size_t>(bh) * Lk * D, out + orow * D);
          }
        }
        __syncwarp();
        st_release_u32(&ep_done[q], s + 1);
      }
    }
  } else {
    // ------------------------------------------------------------ selection
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const bool active = quad < RPU / 32;  // lanes of the MMA tile that belong to the unit
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t acc_it = 0;
    Sel heap;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int bh, qt, part;
      decode(u, bh, qt, part);
      const int i_row = qt * RPU + row;
      if (active) heap.init(sel_mem, row, topk, rec_cap);
      int t0, t1;
      bool empty;
      tile_range(bh, qt, part, t0, t1, empty);
      const uint32_t lim = empty ? 0u : row_limit(bh, i_row);
      const int lim_min = empty ? 0 : tile_limit_min(bh, qt);
      for (int kt = t0; kt < t1; ++kt, ++acc_it) {
        const int b = acc_it % NACC;
        if (!warp_wait(&acc_full[b], (acc_it / NACC) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (!active) {  // no rows of this unit in these lanes: release the accumulator
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);
          continue;
        }
        const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(b * N);
        const uint32_t jt = static_cast<uint32_t>(kt * N);
#pragma unroll 1
        for (int c = 0; c < N / 64; ++c) {
          float vals[64];
          __syncwarp();
          tmem_ld64(taddr + c * 64, vals);
          tmem_wait_ld();
          if (c == N / 64 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
          }
          const uint32_t j0 = jt + static_cast<uint32_t>(c * 64);
          if (static_cast<int>(j0) + 64 > lim_min) mask_scores(vals, j0, lim);
          constexpr int OW = L::OW;
#pragma unroll
          for (int h = 0; h < 64 / OW; ++h)
            heap.offer(reinterpret_cast<const float(&)[OW]>(vals[h * OW]), j0 + static_cast<uint32_t>(h * OW));
        }
      }
      if (!ok) break;
      if (!active) continue;
      heap.finish();  // every lane takes part (warp-synchronous flush)
      if (i_row < Lq && parts > 1) {  // this part's kept keys, for the merge
        const size_t prow = static_cast<size_t>(part) * BH * Lq + static_cast<size_t>(bh) * Lq + i_row;
        for (int t = 0; t < heap.n; ++t) part_keys[prow * topk + t] = heap.get(t);
        part_n[prow] = heap.n;
      } else if (i_row < Lq) {
        const size_t orow = static_cast<size_t>(bh) * Lq + i_row;
        softmax_gather_store<__nv_bfloat16, D>(heap, v + static_cast<size_t>(bh) * Lk * D, out + orow * D);
        if (idx || score)
          write_selection(heap, idx ? idx + orow * topk : nullptr, score ? score + orow * topk : nullptr);
      }
      __syncwarp();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// Key parts per query tile: split only grids that would leave at least half
// the SMs idle (a few query tiles against many keys), into as many parts as
// fill the SMs in one wave, each with at least 4 key tiles.
int tc_parts(const AttnArgs& a, int num_sms, int N, int rpu) {
  const long long units = static_cast<long long>(a.B) * a.H * ((a.Lq + rpu - 1) / rpu);
  if (units * 2 > num_sms) return 1;
  const int kend_min = a.causal ? std::min(a.Lk, rpu + (a.Lk - a.Lq)) : a.Lk;  // query tile 0's key range
  const int nk_min = (kend_min + N - 1) / N;
  long long p = num_sms / units;
  p = std::min<long long>(p, nk_min / 4);
  p = std::min<long long>(p, 8);
  return static_cast<int>(std::max<long long>(p, 1));
}

size_t parts_bytes(const AttnArgs& a, int parts) {
  if (parts <= 1) return 0;
  const size_t rows = static_cast<size_t>(a.B) * a.H * a.Lq;
  return static_cast<size_t>(parts) * rows * (static_cast<size_t>(a.topk) * 8 + 4);
}

constexpr int kMergeWarps = 8;

// Merges a row's `parts` kept lists (each the exact top k of its key range,
// so the union holds the row's top k): one warp per row sorts the packed keys
// (descending, a bitonic network in shared memory; empty slots are 0, below
// every key), keeps the first k, applies the softmax over them and gathers
// their value rows (each lane D / 32 columns).  Writes the selection too if
// asked, in the same order as the single-pass kernel.
template <int D>
__global__ void __launch_bounds__(kMergeWarps * 32)
    attn_merge_kernel(const uint64_t* __restrict__ part_keys, const int* __restrict__ part_n, int parts, int BH,
                      int Lq, int Lk, int topk, int P2, const __nv_bfloat16* __restrict__ v,
                      __nv_bfloat16* __restrict__ out, int32_t* __restrict__ idx, float* __restrict__ score) {
  extern __shared__ uint64_t mk_all[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t* mk = mk_all + static_cast<size_t>(warp) * P2;
  const long long rows = static_cast<long long>(BH) * Lq;
  constexpr int CPL = D / 32;  // columns per lane
  for (long long r = static_cast<long long>(blockIdx.x) * kMergeWarps + warp; r < rows;
       r += static_cast<long long>(gridDim.x) * kMergeWarps) {
    for (int p = 0; p < parts; ++p) {
      const long long pr = static_cast<long long>(p) * rows + r;
      // counts and keys are checked before use: after a kernel that stopped
      // early (a wait ran out) they may never have been written
      const int n = min(max(__ldg(part_n + pr), 0), topk);
      for (int t = lane; t < topk; t += 32) {
        uint64_t key = t < n ? __ldg(reinterpret_cast<const unsigned long long*>(part_keys) + pr * topk + t) : 0ull;
        if (key_index(key) >= static_cast<uint32_t>(Lk)) key = 0ull;
        mk[p * topk + t] = key;
      }
    }
    for (int t = parts * topk + lane; t < P2; t += 32) mk[t] = 0ull;
    __syncwarp();
    for (int kk = 2; kk <= P2; kk <<= 1)
      for (int j = kk >> 1; j > 0; j >>= 1) {
        for (int i = lane; i < P2; i += 32) {
          const int ixj = i ^ j;
          if (ixj > i) {
            const uint64_t x = mk[i], y = mk[ixj];
            const bool down = (i & kk) == 0;  // this half sorts descending
            if (down ? (x < y) : (x > y)) {
              mk[i] = y;
              mk[ixj] = x;
            }
          }
        }
        __syncwarp();
      }
    int keep = 0;  // nonzero keys sort first
    for (int t = lane; t < topk; t += 32) keep += mk[t] != 0ull ? 1 : 0;
    keep = __reduce_add_sync(0xffffffffu, static_cast<unsigned>(keep));
    const int bh = static_cast<int>(r / Lq);
    float acc[CPL];
#pragma unroll
    for (int e = 0; e < CPL; ++e) acc[e] = 0.f;
    float z = 0.f;
    if (keep > 0) {
      const float m = key_score(mk[0]);
      const __nv_bfloat16* vb = v + static_cast<size_t>(bh) * Lk * D + lane * CPL;
      for (int t = 0; t < keep; ++t) {
        const uint64_t key = mk[t];
        const float w = expf(key_score(key) - m);
        z += w;
        const __nv_bfloat16* vr = vb + static_cast<size_t>(key_index(key)) * D;
        if constexpr (CPL == 2) {
          const uint32_t u = __ldg(reinterpret_cast<const unsigned int*>(vr));
          acc[0] = fmaf(w, __uint_as_float(u << 16), acc[0]);
          acc[1] = fmaf(w, __uint_as_float(u & 0xffff0000u), acc[1]);
        } else {
          const uint2 u = __ldg(reinterpret_cast<const uint2*>(vr));
          acc[0] = fmaf(w, __uint_as_float(u.x << 16), acc[0]);
          acc[1] = fmaf(w, __uint_as_float(u.x & 0xffff0000u), acc[1]);
          acc[2] = fmaf(w, __uint_as_float(u.y << 16), acc[2]);
          acc[3] = fmaf(w, __uint_as_float(u.y & 0xffff0000u), acc[3]);
        }
      }
    }
    const float inv = keep > 0 ? 1.f / z : 0.f;
    __nv_bfloat16* orow = out + static_cast<size_t>(r) * D + lane * CPL;
#pragma unroll
    for (int e = 0; e < CPL; e += 2) {
      __nv_bfloat162 h = __floats2bfloat162_rn(acc[e] * inv, acc[e + 1] * inv);
      *reinterpret_cast<__nv_bfloat162*>(orow + e) = h;
    }
    if (idx || score)
      for (int t = lane; t < topk; t += 32) {
        const bool have = t < keep;
        if (idx) idx[static_cast<size_t>(r) * topk + t] = have ? static_cast<int32_t>(key_index(mk[t])) : -1;
        if (score) score[static_cast<size_t>(r) * topk + t] = have ? key_score(mk[t]) : -INFINITY;
      }
    __syncwarp();
  }
}

template <int D, int FK, bool SPLIT, int RPU = BM>
int launch_tc_k(const AttnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  using L = Layout<D, FK, SPLIT, RPU>;
  const int BH = a.B * a.H;
  CUtensorMap tmq, tmk;
  if (!make_tmap_bf16_3d(&tmq, a.q, D, a.Lq, BH, BM)) return -1;
  if (!make_tmap_bf16_3d(&tmk, a.k, D, a.Lk, BH, L::N)) return -1;
  const int parts = tc_parts(a, num_sms, L::N, RPU);
  const int n_units = BH * ((a.Lq + RPU - 1) / RPU) * parts;
  // At least 120 KB so that a second CTA never shares the SM: each CTA takes
  // all TMEM columns it needs for its whole (persistent) lifetime.
  const size_t need = L::bytes(a.topk);
  const size_t smem = need > 120 * 1024 ? need : 120 * 1024;
  auto kern = attn_tc_kernel<D, FK, SPLIT, RPU>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
      cudaSuccess)
    return -1;
  const int grid = n_units < num_sms ? n_units : num_sms;
  const size_t pbytes = SPLIT ? park_bytes(grid, a.topk) : 0;
  if (!a.workspace || a.workspace_bytes < pbytes + parts_bytes(a, parts)) {
    if (SPLIT || parts > 1) return -1;
  }
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  uint64_t* park = nullptr;
  int* park_n = nullptr;
  if constexpr (SPLIT) {
    park = reinterpret_cast<uint64_t*>(ws);
    park_n = reinterpret_cast<int*>(park + static_cast<size_t>(grid) * park_keys_per_cta(a.topk));
  }
  uint64_t* part_keys = nullptr;
  int* part_n = nullptr;
  if (parts > 1) {
    const size_t rows = static_cast<size_t>(BH) * a.Lq;
    part_keys = reinterpret_cast<uint64_t*>(ws + pbytes);
    part_n = reinterpret_cast<int*>(part_keys + static_cast<size_t>(parts) * rows * a.topk);
    // counts start at 0, so that rows a stopped kernel never reached merge as empty
    if (cudaMemsetAsync(part_n, 0, static_cast<size_t>(parts) * rows * sizeof(int), st) != cudaSuccess) return -1;
  }
  kern<<<grid, kThreads<SPLIT>, smem, st>>>(tmq, tmk, static_cast<const __nv_bfloat16*>(a.v),
                                            static_cast<__nv_bfloat16*>(a.out), BH, a.H, a.Lq, a.Lk, a.topk,
                                            L::cap(a.topk), a.causal, a.kv_len, n_units, parts, part_keys, part_n,
                                            parts > 1 ? nullptr : a.idx, parts > 1 ? nullptr : a.score, park,
                                            park_n, ctl);
  if (cudaGetLastError() != cudaSuccess) return -1;
  if (parts == 1) return 1;
  int P2 = 32;
  while (P2 < parts * a.topk) P2 <<= 1;
  const size_t msmem = static_cast<size_t>(kMergeWarps) * P2 * 8;
  auto merge = attn_merge_kernel<D>;
  if (msmem > 48 * 1024 &&
      cudaFuncSetAttribute(merge, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(msmem)) != cudaSuccess)
    return -1;
  const long long rows = static_cast<long long>(BH) * a.Lq;
  long long mgrid = (rows + kMergeWarps - 1) / kMergeWarps;
  if (mgrid > 16LL * num_sms) mgrid = 16LL * num_sms;
  merge<<<static_cast<unsigned>(mgrid), kMergeWarps * 32, msmem, st>>>(
      part_keys, part_n, parts, BH, a.Lq, a.Lk, a.topk, P2, static_cast<const __nv_bfloat16*>(a.v),
      static_cast<__nv_bfloat16*>(a.out), a.idx, a.score);
  return cudaGetLastError() == cudaSuccess ? 2 : -1;
}

// Which kernel serves a shape: the split selection where its heaps and rings
// fit, else the single-warp kernel; fixed heap shapes: 8-ary for k = 64,
// two-level (8 x 16) for 65 <= k <= 137.
// and, for k above what 128 rows' heaps can hold, the single-warp kernel on
// units of 64 (k <= 256) or 32 (k <= 512) query rows.
enum class TcKind { Split64, Split128, Split0, Single64, Single128, Single0, Single0R64, Single0R32 };

template <int D>
TcKind pick(int topk) {
  const bool two_level = topk >= 65 && topk <= 137;
  if (topk == 64 && Layout<D, 64, true>::fits(64)) return TcKind::Split64;
  if (two_level && Layout<D, 128, true>::fits(topk)) return TcKind::Split128;
  if (Layout<D, 0, true>::fits(topk)) return TcKind::Split0;
  if (topk == 64 && Layout<D, 64, false>::fits(64)) return TcKind::Single64;
  if (two_level && Layout<D, 128, false>::fits(topk)) return TcKind::Single128;
  if (Layout<D, 0, false>::fits(topk)) return TcKind::Single0;
  if (topk <= 256 && Layout<D, 0, false, 64>::fits(topk)) return TcKind::Single0R64;
  return TcKind::Single0R32;
}

int rows_per_unit(TcKind k) { return k == TcKind::Single0R64 ? 64 : (k == TcKind::Single0R32 ? 32 : BM); }

bool is_split(TcKind k) { return k == TcKind::Split64 || k == TcKind::Split128 || k == TcKind::Split0; }

template <int D>
int launch_tc(const AttnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  switch (pick<D>(a.topk)) {
    case TcKind::Split64: return launch_tc_k<D, 64, true>(a, ctl, num_sms, st);
    case TcKind::Split128: return launch_tc_k<D, 128, true>(a, ctl, num_sms, st);
    case TcKind::Split0: return launch_tc_k<D, 0, true>(a, ctl, num_sms, st);
    case TcKind::Single64: return launch_tc_k<D, 64, false>(a, ctl, num_sms, st);
    case TcKind::Single128: return launch_tc_k<D, 128, false>(a, ctl, num_sms, st);
    case TcKind::Single0R64: return launch_tc_k<D, 0, false, 64>(a, ctl, num_sms, st);
    case TcKind::Single0R32: return launch_tc_k<D, 0, false, 32>(a, ctl, num_sms, st);
    default: return launch_tc_k<D, 0, false>(a, ctl, num_sms, st);
  }
}

}  // namespace

// Whether the kernel pick() chooses fits in shared memory.
template <int D>
bool tc_fits(int topk) {
  switch (pick<D>(topk)) {
    case TcKind::Split64: return Layout<D, 64, true>::fits(topk);
    case TcKind::Split128: return Layout<D, 128, true>::fits(topk);
    case TcKind::Split0: return Layout<D, 0, true>::fits(topk);
    case TcKind::Single64: return Layout<D, 64, false>::fits(topk);
    case TcKind::Single128: return Layout<D, 128, false>::fits(topk);
    case TcKind::Single0R64: return Layout<D, 0, false, 64>::fits(topk);
    case TcKind::Single0R32: return Layout<D, 0, false, 32>::fits(topk);
    default: return Layout<D, 0, false>::fits(topk);
  }
}

bool attn_tc_supports(const AttnArgs& a) {
  if (a.dtype != 1 || a.topk > kTcMaxK || a.mask) return false;  // bit masks run on the SIMT kernel
  if (a.d == 64) return tc_fits<64>(a.topk);
  if (a.d == 128) return tc_fits<128>(a.topk);
  return false;
}

size_t attn_tc_workspace_bytes(const AttnArgs& a, int num_sms) {
  if (!attn_tc_supports(a)) return 0;
  const TcKind kind = a.d == 64 ? pick<64>(a.topk) : pick<128>(a.topk);
  const int N = a.d == 64 ? (is_split(kind) ? TcShape<64, true>::N : TcShape<64, false>::N) : TcShape<128, true>::N;
  const int rpu = rows_per_unit(kind);
  const int parts = tc_parts(a, num_sms, N, rpu);
  const long long n_units = static_cast<long long>(a.B) * a.H * ((a.Lq + rpu - 1) / rpu) * parts;
  const int grid = n_units < num_sms ? static_cast<int>(n_units) : num_sms;
  return (is_split(kind) ? park_bytes(grid, a.topk) : 0) + parts_bytes(a, parts);
}

int attn_tc(const AttnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  if (!attn_tc_supports(a)) return 0;
  return a.d == 64 ? launch_tc<64>(a, ctl, num_sms, st) : launch_tc<128>(a, ctl, num_sms, st);
}

}  // namespace topk
