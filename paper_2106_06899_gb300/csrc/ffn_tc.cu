// ffn_tc.cu -- top-k feed-forward layer (Eq. 3 with the top-k of Eq. 4) for
// bf16 inputs on sm_103a.
//
// Keys and values are the rows of W1 and W2 (Sec. 2.1), so a token x_i keeps
// the k largest scores s_ij = x_i . W1_j over all d_ff keys, applies ReLU to
// them and sums the matching rows of W2.  Three kernels:
//
// 1. ffn_score_select_kernel (persistent, one CTA per SM).  A work unit is a
//    128-token tile x one slice of the d_ff keys.  TMA streams x and W1
//    chunks of 64 columns; tcgen05.mma accumulates the [128 x 256] score
//    tile in TMEM (double buffered); thread t of the selection warps owns
//    token row t.  Each row keeps a lower bound L of its slice's k-th
//    largest score and appends a score s to its candidate list for this
//    slice (device workspace, linear in tokens) only if s > L and s >= Lg,
//    Lg being the row's bound shared across slices.  L comes from a 64-bin
//    histogram of the candidates' scores kept in shared memory: the lower
//    edge of the highest bin with k candidates at or above it is <= the
//    k-th largest score.  Keys of a slice stream in ascending index order,
//    so the k candidates behind L all have lower indices than any key still
//    to come: a later key scoring exactly L ranks below all of them (ties go
//    to the lower index) and is not appended.  A row of equal scores (an
//    all-zero token, say) thus keeps about k candidates per slice, not all
//    of its keys.  Rows share a bound across slices through one word per
//    row (the k-th largest of any subset of keys is <= that of all keys);
//    its supporting keys may sit in other slices, at higher indices, so it
//    is applied non-strictly.  When bound filtering cannot free room in a
//    list, the list is compacted exactly to its k best entries and L rises
//    to the k-th of them (same argument), so no input overflows a list.
// 2. ffn_finalize_kernel (one CTA per token).  Reads the row's candidates
//    from every slice and keeps the exact top-k by the total order (score
//    descending, index ascending), sorted, in the workspace.
// 3. ffn_gather_kernel (one CTA per column chunk and token, chunk-major).
//    Applies ReLU and gathers the W2 rows with fp32 accumulation.
//
// No [tokens x d_ff] score matrix is ever written to device memory.
#include <algorithm>

#include "kernels.h"
#include "select.cuh"

namespace topk {

namespace {

constexpr int BM = 128;   // tokens per tile
constexpr int NT = 256;   // keys per tile (MMA N)
constexpr int KC = 64;    // d_model columns per pipeline stage
constexpr int S = 3;      // pipeline stages
constexpr int kThreads = 192;
constexpr int NBINS = 64;
constexpr uint32_t A_BYTES = BM * KC * 2;  // 16 KB
constexpr uint32_t B_BYTES = NT * KC * 2;  // 32 KB
constexpr uint32_t ST_BYTES = A_BYTES + B_BYTES;
constexpr int GR = 10;    // pending score groups per row (a 64-score call adds up to 8)
constexpr size_t OFF_HIST = static_cast<size_t>(S) * ST_BYTES;
constexpr size_t OFF_REC = OFF_HIST + static_cast<size_t>(NBINS) * BM * 4;
constexpr size_t OFF_CTRL = OFF_REC + static_cast<size_t>(GR) * BM * 36;
constexpr size_t SMEM_A = 1024 + OFF_CTRL + 256;

constexpr int kFinalThreads = 256;
constexpr int kFinalMaxCand = 8192;  // candidates at or above the final bound held in shared memory
constexpr int kFinalVec = 4;         // 16-byte candidate vectors each finalize thread loads per step

struct Plan {
  int n_rt, tiles, n_sl, n_units, cap;
  size_t off_cnt, off_tau, off_part, off_kept, bytes;
};

Plan make_plan(int N, int d_model, int d_ff, int topk, int num_sms) {
  (void)d_model;
  Plan p{};
  p.n_rt = (N + BM - 1) / BM;
  p.tiles = (d_ff + NT - 1) / NT;
  // slices: minimise waves x tiles-per-slice, plus a small charge per slice.
  // Each slice bounds only its own k-th score, so a slice keeps about
  // k (1 + ln(slice/k)) candidates per row: slices are kept at >= 32 k keys
  // (unless that leaves fewer units than SMs / 4) to hold that volume down.
  double best = 1e30;
  int max_sl = std::max(1, std::min(p.tiles, 64));
  const int by_k = std::max(1, d_ff / (32 * std::max(topk, 1)));
  if (by_k < max_sl && static_cast<long>(p.n_rt) * by_k * 4 >= num_sms) max_sl = by_k;
  for (int sl = 1; sl <= max_sl; ++sl) {
    const long units = static_cast<long>(p.n_rt) * sl;
    const long waves = (units + num_sms - 1) / num_sms;
    const long per = (p.tiles + sl - 1) / sl;
    const double cost = static_cast<double>(waves * per) + 0.5 * sl;
    if (cost < best - 1e-9) {
      best = cost;
      p.n_sl = sl;
    }
  }
  p.n_units = p.n_rt * p.n_sl;
  const int slice_keys = ((p.tiles + p.n_sl - 1) / p.n_sl) * NT;
  // room for about k (1 + ln(slice/k)) candidates plus the bound's lag,
  // so that the in-place compaction (a slow path) stays rare
  const int want = 6 * topk + 1024;
  p.cap = ((std::min(slice_keys, want) + 63) / 64) * 64;
  const size_t rows_sl = static_cast<size_t>(N) * p.n_sl;
  p.off_cnt = rows_sl * p.cap * sizeof(uint2);
  p.off_tau = p.off_cnt + rows_sl * sizeof(int);
  p.off_part = p.off_tau + static_cast<size_t>(N) * sizeof(uint32_t);
  p.off_kept = (p.off_part + rows_sl * sizeof(uint32_t) + 15) & ~size_t(15);
  p.bytes = p.off_kept + static_cast<size_t>(N) * topk * sizeof(uint64_t);  // kept keys per token
  return p;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, const DevCtl& ctl,
                                          volatile int* abort_flag) {
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ctl, abort_flag) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity, const DevCtl& ctl) {
  const unsigned long long t0 = global_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_ns() - t0 > ctl.wait_limit_ns) {
      atomicOr(ctl.error, kDevErrTimeout);
      return;
    }
  }
}

// Per-row candidate state of the selection threads.
//
// The histogram bins are linear in the score value: bin b counts candidates
// with (s - base) / width in [b, b+1), the last bin everything above.  The
// bound derived from bin b is taken one bin lower (base + (b-1) width), so
// that fp32 rounding of the bin index can never place a candidate above
// the bound it supports.
struct RowCand {
  uint2* list;        // this (row, slice)'s candidate list, ascending key index
  uint32_t* hist;     // &hist[bin 0][row], stride BM
  int cap, cnt, k;
  bool hist_on;
  float base, width, inv_width;
  float L;            // this slice already holds k keys scoring >= L, all of lower index than
                      // any key still to come: a later key must beat L strictly
  float mn, mx;       // spread of the first k candidates
  int kp;             // ceil(k / slices)
  float Lp;           // valid lower bound of this slice's kp-th largest score

  __device__ __forceinline__ int bin(float s) const {
    const float f = fminf((s - base) * inv_width, static_cast<float>(NBINS - 1));
    return f > 0.0f ? static_cast<int>(f) : 0;
  }

  __device__ __forceinline__ void add(float s, uint32_t j) {
    if (cnt < cap) list[cnt] = make_uint2(__float_as_uint(s), j);
    ++cnt;
    if (hist_on) {
      hist[bin(s) * BM] += 1u;
    } else {
      mn = fminf(mn, s);
      mx = fmaxf(mx, s);
    }
  }

  // Raise L from the histogram (called between key tiles).
  __device__ __forceinline__ void refresh() {
    if (!hist_on) {
      if (cnt < k) return;
      // at least k candidates so far, every one of them >= mn
      L = fmaxf(L, mn);
      base = mn;
      width = fmaxf((mx - mn) * (1.0f / 48.0f), fmaxf(fabsf(mx), 1e-20f) * 1e-6f);
      inv_width = 1.0f / width;
      hist[0] = static_cast<uint32_t>(cnt - 1);
      hist[bin(mx) * BM] += 1u;
      hist_on = true;
      return;
    }
    // scan from the top bin down, eight bins per step: the eight loads are
    // independent, so their latencies overlap
    uint32_t acc = 0;
    int bstar = 0, bpart = -1;
    for (int b0 = NBINS - 8; b0 >= 0; b0 -= 8) {
      uint32_t h8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) h8[i] = hist[(b0 + i) * BM];
      bool done = false;
#pragma unroll
      for (int i = 7; i >= 0; --i) {
        if (done) continue;
        acc += h8[i];
        if (bpart < 0 && acc >= static_cast<uint32_t>(kp)) bpart = b0 + i;  // kp <= k: found first
        if (acc >= static_cast<uint32_t>(k)) {
          bstar = b0 + i;
          done = true;
        }
      }
      if (done) break;
    }
    if (bpart >= 2) Lp = fmaxf(Lp, base + static_cast<float>(bpart - 1) * width);
    if (bstar >= 2) {
      L = fmaxf(L, base + static_cast<float>(bstar - 1) * width);
      if (bstar >= NBINS / 2) {  // slide the window up: read every bin, then write
        const int sh = bstar - 1;
        uint32_t h[NBINS];
#pragma unroll
        for (int b = 0; b < NBINS; ++b) h[b] = b + sh < NBINS ? hist[(b + sh) * BM] : 0u;
#pragma unroll
        for (int b = 0; b < NBINS; ++b) hist[b * BM] = h[b];
        base += static_cast<float>(sh) * width;
      }
    }
  }

  // Pending score groups ([slot][row] records: 8 scores and the first key).
  float4* rlo;
  float4* rhi;
  uint32_t* rj;
  int rc;

  // A score qualifies for the list if it reaches the shared bound Lg and
  // beats the slice's own bound Ls strictly (see L above).
  __device__ __forceinline__ static bool keep(float s, float Lg, float Ls) { return s >= Lg && s > Ls; }

  // Expand every lane's records into its candidate list, lanes in lockstep:
  // per record slot each lane forms the mask of its qualifying elements,
  // then the warp appends one element per lane per step.
  __device__ __forceinline__ void flush(float Lg, float Ls, bool active) {
    const int mxr = __reduce_max_sync(0xffffffffu, static_cast<unsigned>(active ? rc : 0));
    for (int i = 0; i < mxr; ++i) {
      unsigned msk = 0;
      uint32_t j0 = 0;
      if (active && i < rc) {
        const float4 a = rlo[i * BM];
        const float4 b = rhi[i * BM];
        j0 = rj[i * BM];
        msk = (keep(a.x, Lg, Ls) ? 1u : 0u) | (keep(a.y, Lg, Ls) ? 2u : 0u) | (keep(a.z, Lg, Ls) ? 4u : 0u) |
              (keep(a.w, Lg, Ls) ? 8u : 0u) | (keep(b.x, Lg, Ls) ? 16u : 0u) | (keep(b.y, Lg, Ls) ? 32u : 0u) |
              (keep(b.z, Lg, Ls) ? 64u : 0u) | (keep(b.w, Lg, Ls) ? 128u : 0u);
      }
      while (__any_sync(0xffffffffu, msk != 0)) {
        if (msk) {
          const int e = __ffs(msk) - 1;
          msk &= msk - 1;
          const float v = e < 4 ? reinterpret_cast<const float*>(rlo + i * BM)[e]
                                : reinterpret_cast<const float*>(rhi + i * BM)[e - 4];
          add(v, j0 + e);
        }
      }
    }
    rc = 0;
  }

  // Offer 64 scores (key indices j0..j0+63): each group of 8 whose maximum
  // qualifies (keep()) becomes one record (NaN, used for keys past d_ff,
  // never does).
  __device__ __forceinline__ void offer64(const float (&v)[64], uint32_t j0, float Lg, float Ls, bool active) {
    float m[8];
#pragma unroll
    for (int g = 0; g < 8; ++g)
      m[g] = max3f(max3f(v[8 * g], v[8 * g + 1], v[8 * g + 2]), max3f(v[8 * g + 3], v[8 * g + 4], v[8 * g + 5]),
                   fmaxf(v[8 * g + 6], v[8 * g + 7]));
    if (active) {
      int r = rc;
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        if (keep(m[g], Lg, Ls)) {
          rlo[r * BM] = make_float4(v[8 * g], v[8 * g + 1], v[8 * g + 2], v[8 * g + 3]);
          rhi[r * BM] = make_float4(v[8 * g + 4], v[8 * g + 5], v[8 * g + 6], v[8 * g + 7]);
          rj[r * BM] = j0 + 8 * g;
          ++r;
        }
      }
      rc = r;
    }
    if (__any_sync(0xffffffffu, active && rc > GR - 8)) flush(Lg, Ls, active);
  }

  // The list's exact top k by the total order (score descending, index
  // ascending), in place, keeping list order; L rises to the k-th score.
  // Called when filtering by the bound frees too little room (many keys
  // scoring within a histogram bin of the k-th): every dropped entry ranks
  // below k entries of the list, and so does any later key that does not
  // beat L strictly (the k kept entries have lower indices).  Needs cnt > k.
  // The k-th largest score is found bit by bit (MSB first) on the ordered
  // score keys, below the prefix that every entry shares.
  __device__ void compact_exact() {
    uint32_t lo = 0xFFFFFFFFu, hi = 0u;
    for (int i = 0; i < cnt; ++i) {
      const uint32_t o = ord_f32(__uint_as_float(list[i].x));
      lo = min(lo, o);
      hi = max(hi, o);
    }
    uint32_t t = 0;
    if (lo == hi) {
      t = lo;
    } else {
      const int top = 31 - __clz(lo ^ hi);  // highest bit where entries differ
      t = hi & ~((2u << top) - 1u);         // the shared prefix (bit `top` and below cleared)
      for (int b = top; b >= 0; --b) {
        const uint32_t cand = t | (1u << b);
        int c = 0;
        for (int i = 0; i < cnt; ++i) c += ord_f32(__uint_as_float(list[i].x)) >= cand ? 1 : 0;
        if (c >= k) t = cand;
      }
    }
    // t: ordered key of the k-th largest score.  Keep every entry above it and,
    // in list (= index) order, as many entries equal to it as make k.
    int above = 0;
    for (int i = 0; i < cnt; ++i) above += ord_f32(__uint_as_float(list[i].x)) > t ? 1 : 0;
    int eq_left = k - above;
    int w = 0;
    for (int i = 0; i < cnt; ++i) {
      const uint2 e = list[i];
      const uint32_t o = ord_f32(__uint_as_float(e.x));
      const bool take = o > t || (o == t && eq_left > 0);
      if (o == t && take) --eq_left;
      if (take) list[w++] = e;
    }
    cnt = w;
    L = fmaxf(L, unord_f32(t));
  }
};

__global__ void __launch_bounds__(kThreads, 1)
    ffn_score_select_kernel(const __grid_constant__ CUtensorMap tmx, const __grid_constant__ CUtensorMap tmw,
                            int N, int d_model, int d_ff, int topk, int n_rt, int n_sl, int tiles, int n_units,
                            int cap, uint2* __restrict__ cand, int* __restrict__ cand_cnt,
                            uint32_t* __restrict__ row_tau, uint32_t* __restrict__ row_part, DevCtl ctl) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint32_t* hist_mem = reinterpret_cast<uint32_t*>(smem + OFF_HIST);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_CTRL);
  uint64_t* full = bars;
  uint64_t* empty = bars + S;
  uint64_t* acc_full = bars + 2 * S;
  uint64_t* acc_empty = bars + 2 * S + 2;
  uint64_t* drain = bars + 2 * S + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  constexpr uint32_t IDESC = idesc_bf16_f32(BM, NT);
  constexpr uint32_t TMEM_COLS = 2 * NT;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_kc = d_model / KC;

  // unit u: consecutive units share a d_ff slice, so concurrent CTAs read the same W1 rows
  auto decode = [&](int u, int& rt, int& sl) {
    sl = u / n_rt;
    rt = u % n_rt;
  };
  auto slice_tiles = [&](int sl, int& t0, int& t1) {
    t0 = static_cast<int>(static_cast<long>(tiles) * sl / n_sl);
    t1 = static_cast<int>(static_cast<long>(tiles) * (sl + 1) / n_sl);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmx);
      tma_prefetch_desc(&tmw);
    }
    uint32_t it = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int rt, sl, t0, t1;
      decode(u, rt, sl);
      slice_tiles(sl, t0, t1);
      for (int kt = t0; ok && kt < t1; ++kt) {
        for (int kc = 0; kc < n_kc; ++kc) {
          const int s = it % S;
          if (!warp_wait(&empty[s], ((it / S) & 1u) ^ 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            uint8_t* st = smem + static_cast<size_t>(s) * ST_BYTES;
            mbar_arrive_expect_tx(&full[s], ST_BYTES);
            tma_load_2d(st, &tmx, &full[s], kc * KC, rt * BM);
            tma_load_2d(st + A_BYTES, &tmw, &full[s], kc * KC, kt * NT);
          }
          ++it;
        }
      }
    }
    if (lane == 0) {
      for (uint32_t back = 1; back <= static_cast<uint32_t>(S) && back <= it; ++back) {
        const uint32_t t = it - back;
        mbar_drain(&full[t % S], (t / S) & 1u, ctl);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    uint32_t it = 0, acc_it = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int rt, sl, t0, t1;
      decode(u, rt, sl);
      slice_tiles(sl, t0, t1);
      for (int kt = t0; ok && kt < t1; ++kt, ++acc_it) {
        const int b = acc_it & 1;
        if (!warp_wait(&acc_empty[b], ((acc_it >> 1) & 1u) ^ 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int kc = 0; kc < n_kc; ++kc, ++it) {
          const int s = it % S;
          if (!warp_wait(&full[s], (it / S) & 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) {
            const uint32_t aa = smem_u32(smem + static_cast<size_t>(s) * ST_BYTES);
            const uint32_t ba = aa + A_BYTES;
#pragma unroll
            for (int st = 0; st < KC / 16; ++st)
              mma_bf16_ss(tmem_base + static_cast<uint32_t>(b * NT), sdesc_k128(aa + st * 32),
                          sdesc_k128(ba + st * 32), IDESC, (kc > 0 || st > 0) ? 1u : 0u);
            mma_commit(&empty[s]);
            if (kc == n_kc - 1) mma_commit(&acc_full[b]);
          }
          __syncwarp();
        }
      }
    }
    if (lane == 0) {
      mma_commit(drain);
      mbar_drain(drain, 0, ctl);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ selection
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t acc_it = 0;
    bool ok = true;
    RowCand rc;
    rc.hist = hist_mem + row;
    rc.k = topk;
    rc.cap = cap;
    rc.rlo = reinterpret_cast<float4*>(smem + OFF_REC) + row;
    rc.rhi = reinterpret_cast<float4*>(smem + OFF_REC + static_cast<size_t>(GR) * BM * 16) + row;
    rc.rj = reinterpret_cast<uint32_t*>(smem + OFF_REC + static_cast<size_t>(GR) * BM * 32) + row;
    rc.rc = 0;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int rt, sl, t0, t1;
      decode(u, rt, sl);
      slice_tiles(sl, t0, t1);
      const int grow = rt * BM + row;
      const bool row_ok = grow < N;
      const size_t rs = static_cast<size_t>(row_ok ? grow : 0) * n_sl + sl;
      rc.list = cand + rs * cap;
      rc.cnt = 0;
      rc.hist_on = false;
      rc.base = 0.0f;
      rc.width = 1.0f;
      rc.inv_width = 1.0f;
      rc.L = -INFINITY;
      rc.mn = INFINITY;
      rc.mx = -INFINITY;
      rc.kp = (topk + n_sl - 1) / n_sl;
      rc.Lp = -INFINITY;
      uint32_t published = 0, published_part = 0;
      for (int b = 0; b < NBINS; ++b) rc.hist[b * BM] = 0u;

      for (int kt = t0; kt < t1; ++kt, ++acc_it) {
        // the bound shared by the other slices of this row
        const uint32_t shared_key = row_ok ? *reinterpret_cast<volatile uint32_t*>(row_tau + grow) : 0u;
        const float Lg = shared_key ? unord_f32(shared_key) : -INFINITY;
        const float Ls = rc.L;  // refresh() moves it only after this tile's flush
        const int b = acc_it & 1;
        if (!warp_wait(&acc_full[b], (acc_it >> 1) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(b * NT);
#pragma unroll 1
        for (int c = 0; c < NT / 64; ++c) {
          float v[64];
          __syncwarp();
          tmem_ld64(taddr + c * 64, v);
          tmem_wait_ld();
          if (c == NT / 64 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
          }
          const uint32_t j0 = static_cast<uint32_t>(kt * NT + c * 64);
          if (j0 + 64 > static_cast<uint32_t>(d_ff)) {
#pragma unroll
            for (int e = 0; e < 64; ++e)
              if (j0 + e >= static_cast<uint32_t>(d_ff)) v[e] = __uint_as_float(0x7fc00000u);  // NaN: never kept
          }
          rc.offer64(v, j0, Lg, Ls, row_ok);
        }
        // the tile's pending groups go to the list before the bound moves
        if (__any_sync(0xffffffffu, row_ok && rc.rc > 0)) rc.flush(Lg, Ls, row_ok);
        if (!row_ok) continue;
        rc.refresh();
        const uint32_t lkey = rc.L > -INFINITY ? ord_f32(rc.L) : 0u;
        if (lkey > published) {
          atomicMax(row_tau + grow, lkey);
          published = lkey;
        }
        // Pooled bound: every slice s of the row holds at least kp = ceil(k /
        // slices) scores >= its Lp_s, so the row holds at least k scores >=
        // min_s Lp_s, a valid bound of the row's k-th score however few of
        // the row's top k each slice holds.  A slice publishes its Lp when it
        // rises and raises the row's bound to the minimum of what every
        // slice has published (0 = nothing yet; words only grow, so a stale
        // one only makes the minimum smaller).
        const uint32_t pkey = rc.Lp > -INFINITY ? ord_f32(rc.Lp) : 0u;
        if (n_sl > 1 && pkey > published_part) {
          const size_t r0 = static_cast<size_t>(grow) * n_sl;
          atomicMax(row_part + r0 + sl, pkey);
          published_part = pkey;
          uint32_t mn = pkey;
          for (int q = 0; q < n_sl && mn != 0u; ++q)
            if (q != sl) mn = min(mn, *reinterpret_cast<volatile uint32_t*>(row_part + r0 + q));
          if (mn != 0u) atomicMax(row_tau + grow, mn);
        }
        // ---- make room for the next tile (rare): drop candidates below the
        // bound (entries equal to it may be the row's top k and stay); if that
        // is not enough, keep exactly the list's k best.  cap >= k + 2 NT
        // whenever a slice has more keys than cap (make_plan), so either way
        // the next tile's NT keys fit.
        if (kt + 1 < t1 && rc.cnt > rc.cap - NT) {
          const float Lc = fmaxf(rc.L, Lg);
          int w = 0;
          for (int i = 0; i < rc.cnt; ++i) {
            const uint2 e = rc.list[i];
            if (__uint_as_float(e.x) >= Lc) rc.list[w++] = e;
          }
          rc.cnt = w;
          if (w > rc.cap - NT) rc.compact_exact();
        }
      }
      if (!ok) break;
      if (row_ok) cand_cnt[rs] = rc.cnt;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// One CTA per token row: exact top-k among its candidates.
//
// Only candidates >= L (the row's shared bound) can be in the top-k.  An
// MSB-first radix select over their ordered score keys (11, 11 and 10 bits;
// histograms in shared memory, increments aggregated per warp with
// __match_any_sync so that equal digits do not serialise) finds the exact
// k-th largest score t and how many keys scoring t the kept set takes.  When
// more keys score t than that, the tie rule (lower index first) decides:
// a second radix select, over the complemented indices of the keys scoring
// t, finds the index where the kept ties stop.  The kept set -- every key
// above t plus the chosen ties -- is sorted best first with a bitonic sort
// of the packed keys.  When everything at or above the k-th key's first
// digit fits in shared memory, it is collected and sorted there directly.
constexpr int kHistBins = 2048;

__device__ __forceinline__ void warp_hist_add(uint32_t* hist, uint32_t d, bool valid) {
  const unsigned peers = __match_any_sync(0xffffffffu, valid ? d : 0xFFFFFFFFu);
  const int lane = threadIdx.x & 31;
  if (valid && lane == __ffs(peers) - 1) atomicAdd(&hist[d], static_cast<unsigned>(__popc(peers)));
}

// Warp-aggregated append: returns this lane's slot (or -1 if !take).
__device__ __forceinline__ int warp_append(int* counter, bool take) {
  const unsigned bal = __ballot_sync(0xffffffffu, take);
  if (!bal) return -1;
  const int lane = threadIdx.x & 31;
  int base = 0;
  if (lane == __ffs(bal) - 1) base = atomicAdd(counter, __popc(bal));
  base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
  return take ? base + __popc(bal & ((1u << lane) - 1u)) : -1;
}

// Bitonic sort of keys[0, n) in shared memory, descending; slots n .. next
// power of two are padded with 0 (which ranks last).  All threads call it.
__device__ __forceinline__ void bitonic_desc(uint64_t* keys, int n) {
  int m = 1;
  while (m < n) m <<= 1;
  for (int i = n + static_cast<int>(threadIdx.x); i < m; i += blockDim.x) keys[i] = 0ull;
  __syncthreads();
  for (int size = 2; size <= m; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (m >> 1); i += blockDim.x) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const uint64_t a = keys[lo], b = keys[hi];
        if ((a < b) == desc) {
          keys[lo] = b;
          keys[hi] = a;
        }
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(kFinalThreads)
    ffn_finalize_kernel(uint64_t* __restrict__ kept, int topk, int n_sl, int cap, const uint2* __restrict__ cand,
                        const int* __restrict__ cand_cnt, const uint32_t* __restrict__ row_tau,
                        int32_t* __restrict__ idx, float* __restrict__ score, DevCtl ctl) {
  extern __shared__ uint64_t keys[];  // [kFinalMaxCand]; the first kHistBins words double as the histogram
  __shared__ uint32_t csum[kFinalThreads];
  __shared__ int n_keys, bad, sh_digit, sh_above, sh_count;
  uint32_t* hist = reinterpret_cast<uint32_t*>(keys);
  const int row = blockIdx.x;
  const int tid = threadIdx.x;
  if (tid == 0) {
    n_keys = 0;
    bad = 0;
  }
  __syncthreads();
  const uint32_t tk = row_tau[row];
  const float L = tk ? unord_f32(tk) : -INFINITY;
  for (int sl = tid; sl < n_sl; sl += kFinalThreads) {
    const int c = cand_cnt[static_cast<size_t>(row) * n_sl + sl];
    if (c < 0 || c > cap) bad = 1;  // never written: the first kernel stopped early (a timeout)
  }
  __syncthreads();
  if (bad) {
    if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
    return;
  }
  // visit every candidate slot of the row; all threads iterate together.
  // Each thread loads kFinalVec 16-byte vectors (two candidates each) before
  // it visits any of them, so that many loads are in flight per thread (the
  // lists are read from device memory).  A list starts on a 16-byte
  // boundary and has an even capacity, so a vector never leaves its list;
  // entries at or past the count are skipped.
  auto for_each = [&](auto&& f) {
    for (int sl = 0; sl < n_sl; ++sl) {
      const int c = cand_cnt[static_cast<size_t>(row) * n_sl + sl];
      const uint4* lst = reinterpret_cast<const uint4*>(cand + (static_cast<size_t>(row) * n_sl + sl) * cap);
      for (int b0 = 0; b0 < c; b0 += 2 * kFinalVec * kFinalThreads) {
        uint4 w[kFinalVec];
#pragma unroll
        for (int u = 0; u < kFinalVec; ++u) {
          const int i = b0 + 2 * (u * kFinalThreads + tid);
          w[u] = i < c ? lst[i / 2] : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kFinalVec; ++u) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int i = b0 + 2 * (u * kFinalThreads + tid) + h;
            const uint32_t sx = h ? w[u].z : w[u].x, jx = h ? w[u].w : w[u].y;
            const bool valid = i < c && __uint_as_float(sx) >= L;
            f(valid, valid ? ord_f32(__uint_as_float(sx)) : 0u, jx);
          }
        }
      }
    }
  };
  // One MSB-first radix digit: over the candidates with mine(o, j) whose
  // value val(o, j) matches `prefix` on `pmask`, histogram the digit
  // (val >> sh) & dm and find the digit holding the remaining-th largest
  // value.  Sets sh_digit (-1 if fewer than `remaining` such candidates),
  // sh_above (candidates in higher digits) and sh_count (in that digit).
  auto radix_digit = [&](auto&& mine, auto&& val, uint32_t prefix, uint32_t pmask, int sh, uint32_t dm,
                         int remaining) {
    for (int i = tid; i < kHistBins; i += kFinalThreads) hist[i] = 0u;
    __syncthreads();
    for_each([&](bool valid, uint32_t o, uint32_t j) {
      const uint32_t x = val(o, j);
      warp_hist_add(hist, (x >> sh) & dm, valid && mine(o, j) && (x & pmask) == prefix);
    });
    __syncthreads();
    // chunk sums from the top bin down, then one thread locates the digit
    const int nb = static_cast<int>(dm) + 1, per = (nb + kFinalThreads - 1) / kFinalThreads;
    uint32_t cs = 0;
    for (int q = 0; q < per; ++q) {
      const int bin = nb - 1 - (tid * per + q);
      if (bin >= 0) cs += hist[bin];
    }
    csum[tid] = cs;
    __syncthreads();
    if (tid == 0) {
      uint32_t cum = 0;
      int t = 0;
      for (; t < kFinalThreads; ++t) {
        if (cum + csum[t] >= static_cast<uint32_t>(remaining)) break;
        cum += csum[t];
      }
      int digit = -1;
      for (int q = 0; q < per && t < kFinalThreads; ++q) {
        const int bin = nb - 1 - (t * per + q);
        if (bin < 0) break;
        if (cum + hist[bin] >= static_cast<uint32_t>(remaining)) {
          digit = bin;
          break;
        }
        cum += hist[bin];
      }
      sh_digit = digit;
      sh_above = static_cast<int>(cum);
      sh_count = digit >= 0 ? static_cast<int>(hist[digit]) : 0;
    }
    __syncthreads();
  };
  const int shifts[3] = {21, 10, 0};
  const uint32_t dmasks[3] = {0x7FFu, 0x7FFu, 0x3FFu};
  auto any = [](uint32_t, uint32_t) { return true; };
  auto score_of = [](uint32_t o, uint32_t) { return o; };
  // radix select: the k-th largest ordered score among the candidates
  uint32_t prefix = 0, pmask = 0;
  int remaining = topk, n_eq = 0;
  bool direct = false;
#pragma unroll 1
  for (int pass = 0; pass < 3; ++pass) {
    radix_digit(any, score_of, prefix, pmask, shifts[pass], dmasks[pass], remaining);
    const int digit = sh_digit, above = sh_above, count = sh_count;
    if (digit < 0) {  // fewer candidates than k: cannot happen unless the lists are inconsistent
      if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
      return;
    }
    prefix |= static_cast<uint32_t>(digit) << shifts[pass];
    pmask |= dmasks[pass] << shifts[pass];
    remaining -= above;
    n_eq = count;
    const int kept_or_open = (topk - remaining) + count;
    if (pass == 0 && kept_or_open <= kFinalMaxCand) {
      // everything at or above the k-th key's leading 11 bits fits in shared
      // memory: collect it and finish there (one more read of the lists)
      for_each([&](bool valid, uint32_t o, uint32_t j) {
        const int pa = warp_append(&n_keys, valid && (o & pmask) >= prefix);
        if (pa >= 0 && pa < kFinalMaxCand) keys[pa] = (static_cast<uint64_t>(o) << 32) | static_cast<uint64_t>(~j);
      });
      __syncthreads();
      const int nc = n_keys;
      if (nc != kept_or_open || nc < topk) {
        if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
        return;
      }
      bitonic_desc(keys, nc);
      direct = true;  // keys[0 .. topk) are the kept keys, best first
      break;
    }
  }
  if (!direct) {
    // prefix: ordered key t of the k-th largest score; the kept set takes
    // `remaining` of the n_eq keys scoring t, those of lowest index
    const uint32_t thr = prefix;
    uint32_t jsel = 0;  // a key scoring t is kept iff ~index >= jsel
    if (n_eq > remaining) {
      auto is_tie = [thr](uint32_t o, uint32_t) { return o == thr; };
      auto inv_index = [](uint32_t, uint32_t j) { return ~j; };
      uint32_t p2 = 0, m2 = 0;
      int rem2 = remaining;
#pragma unroll 1
      for (int pass = 0; pass < 3; ++pass) {
        radix_digit(is_tie, inv_index, p2, m2, shifts[pass], dmasks[pass], rem2);
        if (sh_digit < 0) {
          if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
          return;
        }
        p2 |= static_cast<uint32_t>(sh_digit) << shifts[pass];
        m2 |= dmasks[pass] << shifts[pass];
        rem2 -= sh_above;
      }
      jsel = p2;  // the remaining-th largest ~index among the ties (indices are distinct)
    }
    __syncthreads();
    if (tid == 0) n_keys = 0;
    __syncthreads();
    for_each([&](bool valid, uint32_t o, uint32_t j) {
      const int pa = warp_append(&n_keys, valid && (o > thr || (o == thr && ~j >= jsel)));
      if (pa >= 0 && pa < topk) keys[pa] = (static_cast<uint64_t>(o) << 32) | static_cast<uint64_t>(~j);
    });
    __syncthreads();
    if (n_keys != topk) {
      if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
      return;
    }
    bitonic_desc(keys, topk);
  }
  // the kept keys, in selection order, for the gather kernel
  for (int t = tid; t < topk; t += kFinalThreads) kept[static_cast<size_t>(row) * topk + t] = keys[t];
  if (idx || score) {
    for (int t = tid; t < topk; t += kFinalThreads) {
      const uint64_t key = keys[t];
      if (idx) idx[static_cast<size_t>(row) * topk + t] = static_cast<int32_t>(key_index(key));
      if (score) score[static_cast<size_t>(row) * topk + t] = key_score(key);
    }
  }
}

// ReLU over the kept scores and the weighted sum of the matching W2 rows
// (fp32).  One CTA per (column chunk, token), chunk-major: all tokens read
// their rows' first kGatherCols columns before any reads the next chunk, so
// that the W2 columns being read (d_ff x kGatherCols bf16, 32 MB at d_ff =
// 65536) stay resident in L2 while every token visits them.  Each thread
// owns 4 columns and keeps 8 rows in flight.
constexpr int kGatherCols = 256;
constexpr int kGatherThreads = kGatherCols / 4;

__global__ void __launch_bounds__(kGatherThreads)
    ffn_gather_kernel(const __nv_bfloat16* __restrict__ W2, float* __restrict__ out, int N, int d_model, int topk,
                      const uint64_t* __restrict__ kept) {
  extern __shared__ uint64_t gkeys[];  // [topk]
  const int row = blockIdx.x % N;
  const int chunk = blockIdx.x / N;
  const int tid = threadIdx.x;
  for (int t = tid; t < topk; t += kGatherThreads) gkeys[t] = kept[static_cast<size_t>(row) * topk + t];
  __syncthreads();
  const int c0 = chunk * kGatherCols + tid * 4;
  if (c0 >= d_model) return;
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  int t = 0;
  for (; t + 8 <= topk; t += 8) {
    uint2 raw[8];
    float w[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint64_t key = gkeys[t + u];
      w[u] = fmaxf(key_score(key), 0.0f);
      raw[u] = __ldg(reinterpret_cast<const uint2*>(W2 + static_cast<size_t>(key_index(key)) * d_model + c0));
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      a0 = fmaf(w[u], __uint_as_float(raw[u].x << 16), a0);
      a1 = fmaf(w[u], __uint_as_float(raw[u].x & 0xFFFF0000u), a1);
      a2 = fmaf(w[u], __uint_as_float(raw[u].y << 16), a2);
      a3 = fmaf(w[u], __uint_as_float(raw[u].y & 0xFFFF0000u), a3);
    }
  }
  for (; t < topk; ++t) {
    const uint64_t key = gkeys[t];
    const float w = fmaxf(key_score(key), 0.0f);
    const uint2 raw = __ldg(reinterpret_cast<const uint2*>(W2 + static_cast<size_t>(key_index(key)) * d_model + c0));
    a0 = fmaf(w, __uint_as_float(raw.x << 16), a0);
    a1 = fmaf(w, __uint_as_float(raw.x & 0xFFFF0000u), a1);
    a2 = fmaf(w, __uint_as_float(raw.y << 16), a2);
    a3 = fmaf(w, __uint_as_float(raw.y & 0xFFFF0000u), a3);
  }
  *reinterpret_cast<float4*>(out + static_cast<size_t>(row) * d_model + c0) = make_float4(a0, a1, a2, a3);
}

bool make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint32_t box1) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {dim0, dim1};
  cuuint64_t strides[1] = {dim0 * 2};
  cuuint32_t box[2] = {64, box1};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int current_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 152;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 152;
  return n;
}

}  // namespace

size_t ffn_workspace_bytes(int N, int d_model, int d_ff, int topk) {
  return make_plan(N, d_model, d_ff, topk, current_sm_count()).bytes;
}

int ffn_tc(const FfnArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  const Plan p = make_plan(a.N, a.d_model, a.d_ff, a.topk, num_sms);
  if (!a.workspace || a.workspace_bytes < p.bytes) return -1;
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  uint2* cand = reinterpret_cast<uint2*>(ws);
  int* cnt = reinterpret_cast<int*>(ws + p.off_cnt);
  uint32_t* tau = reinterpret_cast<uint32_t*>(ws + p.off_tau);
  uint32_t* part = reinterpret_cast<uint32_t*>(ws + p.off_part);
  CUtensorMap tmx, tmw;
  if (!make_tmap_bf16_2d(&tmx, a.x, a.d_model, a.N, BM)) return -1;
  if (!make_tmap_bf16_2d(&tmw, a.W1, a.d_model, a.d_ff, NT)) return -1;
  if (cudaMemsetAsync(tau, 0, static_cast<size_t>(a.N) * sizeof(uint32_t), st) != cudaSuccess) return -1;
  if (cudaMemsetAsync(part, 0, static_cast<size_t>(a.N) * p.n_sl * sizeof(uint32_t), st) != cudaSuccess) return -1;
  // counts start at -1 ("not written"): the finalize reads no list whose count the first kernel did not set
  if (cudaMemsetAsync(cnt, 0xFF, static_cast<size_t>(a.N) * p.n_sl * sizeof(int), st) != cudaSuccess) return -1;
  if (cudaFuncSetAttribute(ffn_score_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(SMEM_A)) != cudaSuccess)
    return -1;
  const int grid = p.n_units < num_sms ? p.n_units : num_sms;
  ffn_score_select_kernel<<<grid, kThreads, SMEM_A, st>>>(tmx, tmw, a.N, a.d_model, a.d_ff, a.topk, p.n_rt, p.n_sl,
                                                           p.tiles, p.n_units, p.cap, cand, cnt, tau, part, ctl);
  if (cudaGetLastError() != cudaSuccess) return -1;
  constexpr size_t kFinalSmem = kFinalMaxCand * sizeof(uint64_t);
  if (cudaFuncSetAttribute(ffn_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kFinalSmem)) != cudaSuccess)
    return -1;
  uint64_t* kept = reinterpret_cast<uint64_t*>(ws + p.off_kept);
  ffn_finalize_kernel<<<a.N, kFinalThreads, kFinalSmem, st>>>(kept, a.topk, p.n_sl, p.cap, cand, cnt, tau, a.idx,
                                                              a.score, ctl);
  if (cudaGetLastError() != cudaSuccess) return -1;
  const int n_chunks = (a.d_model + kGatherCols - 1) / kGatherCols;
  if (a.w2_ready && cudaStreamWaitEvent(st, a.w2_ready, 0) != cudaSuccess) return -1;
  ffn_gather_kernel<<<n_chunks * a.N, kGatherThreads, static_cast<size_t>(a.topk) * sizeof(uint64_t), st>>>(
      static_cast<const __nv_bfloat16*>(a.W2), a.out, a.N, a.d_model, a.topk, kept);
  if (cudaGetLastError() != cudaSuccess) return -1;
  return 3;
}

}  // namespace topk
