// ffn_tc.cu -- top-k feed-forward layer (Eq. 3 with the top-k of Eq. 4) for
// bf16 inputs on sm_103a.
//
// Keys and values are the rows of W1 and W2 (Sec. 2.1), so a token x_i keeps
// the k largest scores s_ij = x_i . W1_j over all d_ff keys, applies ReLU to
// them and sums the matching rows of W2.  Two kernels:
//
// 1. ffn_score_select_kernel (persistent, one CTA per SM).  A work unit is a
//    128-token tile x one slice of the d_ff keys.  TMA streams x and W1
//    chunks of 64 columns; tcgen05.mma accumulates the [128 x 256] score
//    tile in TMEM (double buffered); thread t of the selection warps owns
//    token row t.  Each row keeps a valid lower bound L of its k-th largest
//    score and appends every score s >= L to its candidate list for this
//    slice (device workspace, linear in tokens).  L comes from a 64-bin
//    histogram of the candidates' scores kept in shared memory: the lower
//    edge of the highest bin with k candidates at or above it is <= the
//    k-th largest score, so raising L to it never drops a true top-k key.
//    Rows also share L across slices through one word per row (the k-th
//    largest of any subset of keys is <= that of all keys).
// 2. ffn_finalize_kernel (one CTA per token).  Reads the row's candidates
//    from every slice, keeps the exact top-k by the total order (score
//    descending, index ascending) with a bitonic sort in shared memory,
//    applies ReLU and gathers the W2 rows with fp32 accumulation.
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
constexpr size_t OFF_HIST = static_cast<size_t>(S) * ST_BYTES;
constexpr size_t OFF_CTRL = OFF_HIST + static_cast<size_t>(NBINS) * BM * 4;
constexpr size_t SMEM_A = 1024 + OFF_CTRL + 256;

constexpr int kFinalThreads = 256;
constexpr int kFinalMaxCand = 8192;  // candidates at or above the final bound held in shared memory

struct Plan {
  int n_rt, tiles, n_sl, n_units, cap;
  size_t off_cnt, off_tau, bytes;
};

Plan make_plan(int N, int d_model, int d_ff, int topk, int num_sms) {
  (void)d_model;
  Plan p{};
  p.n_rt = (N + BM - 1) / BM;
  p.tiles = (d_ff + NT - 1) / NT;
  // slices: minimise waves x tiles-per-slice, plus a small charge per slice
  // (each slice has its own warm-up of k candidates)
  double best = 1e30;
  const int max_sl = std::max(1, std::min(p.tiles, 64));
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
  const int want = 4 * topk + 1024;
  p.cap = ((std::min(slice_keys, want) + 63) / 64) * 64;
  const size_t rows_sl = static_cast<size_t>(N) * p.n_sl;
  p.off_cnt = rows_sl * p.cap * sizeof(uint2);
  p.off_tau = p.off_cnt + rows_sl * sizeof(int);
  p.bytes = p.off_tau + static_cast<size_t>(N) * sizeof(uint32_t);
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
  uint2* list;        // this (row, slice)'s candidate list
  uint32_t* hist;     // &hist[bin 0][row], stride BM
  int cap, cnt, k;
  bool dead;          // list overflowed (outputs invalid, error flagged)
  bool hist_on;
  float base, width, inv_width;
  float L;            // valid lower bound of the row's k-th largest score
  float mn, mx;       // spread of the first k candidates

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
    uint32_t acc = 0;
    int bstar = 0;
    for (int b = NBINS - 1; b >= 0; --b) {
      acc += hist[b * BM];
      if (acc >= static_cast<uint32_t>(k)) {
        bstar = b;
        break;
      }
    }
    if (bstar >= 2) {
      L = fmaxf(L, base + static_cast<float>(bstar - 1) * width);
      if (bstar >= NBINS / 2) {  // slide the window up
        const int sh = bstar - 1;
        for (int b = 0; b < NBINS; ++b) hist[b * BM] = b + sh < NBINS ? hist[(b + sh) * BM] : 0u;
        base += static_cast<float>(sh) * width;
      }
    }
  }
};

__global__ void __launch_bounds__(kThreads, 1)
    ffn_score_select_kernel(const __grid_constant__ CUtensorMap tmx, const __grid_constant__ CUtensorMap tmw,
                            int N, int d_model, int d_ff, int topk, int n_rt, int n_sl, int tiles, int n_units,
                            int cap, uint2* __restrict__ cand, int* __restrict__ cand_cnt,
                            uint32_t* __restrict__ row_tau, DevCtl ctl) {
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
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int rt, sl, t0, t1;
      decode(u, rt, sl);
      slice_tiles(sl, t0, t1);
      const int grow = rt * BM + row;
      const bool row_ok = grow < N;
      const size_t rs = static_cast<size_t>(row_ok ? grow : 0) * n_sl + sl;
      rc.list = cand + rs * cap;
      rc.cnt = 0;
      rc.dead = false;
      rc.hist_on = false;
      rc.base = 0.0f;
      rc.width = 1.0f;
      rc.inv_width = 1.0f;
      rc.L = -INFINITY;
      rc.mn = INFINITY;
      rc.mx = -INFINITY;
      uint32_t published = 0;
      for (int b = 0; b < NBINS; ++b) rc.hist[b * BM] = 0u;

      for (int kt = t0; kt < t1; ++kt, ++acc_it) {
        // the bound shared by the other slices of this row
        const uint32_t shared_key = row_ok ? *reinterpret_cast<volatile uint32_t*>(row_tau + grow) : 0u;
        const float Lg = shared_key ? unord_f32(shared_key) : -INFINITY;
        const float L = fmaxf(rc.L, Lg);
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
          if (row_ok && !rc.dead) {
#pragma unroll
            for (int g = 0; g < 8; ++g) {
              const float* w = &v[8 * g];
              const float m = max3f(max3f(w[0], w[1], w[2]), max3f(w[3], w[4], w[5]), fmaxf(w[6], w[7]));
              if (m >= L) {
#pragma unroll
                for (int e = 0; e < 8; ++e)
                  if (w[e] >= L) rc.add(w[e], j0 + 8 * g + e);
              }
            }
          }
        }
        if (!row_ok || rc.dead) continue;
        rc.refresh();
        const uint32_t lkey = rc.L > -INFINITY ? ord_f32(rc.L) : 0u;
        if (lkey > published) {
          atomicMax(row_tau + grow, lkey);
          published = lkey;
        }
        // ---- make room for the next tile: drop candidates below the bound (rare)
        if (kt + 1 < t1 && rc.cnt > rc.cap - NT) {
          const float Lc = fmaxf(rc.L, Lg);
          int w = 0;
          for (int i = 0; i < rc.cnt; ++i) {
            const uint2 e = rc.list[i];
            if (__uint_as_float(e.x) >= Lc) rc.list[w++] = e;
          }
          rc.cnt = w;
          if (w > rc.cap - NT) {
            rc.dead = true;
            atomicOr(ctl.error, kDevErrWorkspace);
          }
        }
      }
      if (!ok) break;
      if (row_ok) cand_cnt[rs] = rc.dead ? -1 : min(rc.cnt, rc.cap);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// One CTA per token row: exact top-k among its candidates, ReLU, W2 gather.
//
// Only candidates >= L (the row's shared bound) can be in the top-k.  If
// more of them than fit in shared memory remain, an MSB-first radix pass
// over the ordered score keys (8 bits at a time, counted in shared memory)
// narrows the set: after each pass, every key whose leading bits exceed the
// chosen prefix is certainly kept, and those equal to it are still open;
// once kept + open fits, all of them are collected.  The exact top-k is
// then a bitonic sort of the packed keys (score descending, index
// ascending).
__global__ void __launch_bounds__(kFinalThreads)
    ffn_finalize_kernel(const __nv_bfloat16* __restrict__ W2, float* __restrict__ out, int d_model, int topk,
                        int n_sl, int cap, const uint2* __restrict__ cand, const int* __restrict__ cand_cnt,
                        const uint32_t* __restrict__ row_tau, int32_t* __restrict__ idx,
                        float* __restrict__ score, DevCtl ctl) {
  extern __shared__ uint64_t keys[];  // [kFinalMaxCand]
  __shared__ uint32_t hist[256];
  __shared__ int n_keys, bad, sh_digit, sh_above;
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
    if (c < 0 || c > cap) bad = 1;  // overflowed, or never written (first kernel stopped early)
  }
  __syncthreads();
  if (bad) {
    if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
    return;
  }
  // visit every candidate of the row that is >= L: f(ord, index)
  auto for_each = [&](auto&& f) {
    for (int sl = 0; sl < n_sl; ++sl) {
      const int c = cand_cnt[static_cast<size_t>(row) * n_sl + sl];
      const uint2* lst = cand + (static_cast<size_t>(row) * n_sl + sl) * cap;
      for (int i = tid; i < c; i += kFinalThreads) {
        const uint2 e = lst[i];
        const float sc = __uint_as_float(e.x);
        if (sc >= L) f(ord_f32(sc), e.y);
      }
    }
  };
  // radix narrowing: keys with (ord >> (32 - plen)) > prefix are kept for sure
  uint32_t prefix = 0;
  int plen = 0, remaining = topk, total = 0;
  for (;;) {
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    if (plen == 32) break;
    const int shift = 24 - plen;
    for_each([&](uint32_t o, uint32_t) {
      if (plen == 0 || (o >> (32 - plen)) == prefix) atomicAdd(&hist[(o >> shift) & 255u], 1u);
    });
    __syncthreads();
    if (tid == 0) {
      uint32_t cum = 0;
      int d = 255;
      for (; d > 0; --d) {
        if (cum + hist[d] >= static_cast<uint32_t>(remaining)) break;
        cum += hist[d];
      }
      sh_digit = d;
      sh_above = static_cast<int>(cum);
    }
    __syncthreads();
    const int d = sh_digit;
    const int above = sh_above;
    const int open = static_cast<int>(hist[d]);
    prefix = (prefix << 8) | static_cast<uint32_t>(d);
    plen += 8;
    remaining -= above;
    total = (topk - remaining) + open;
    __syncthreads();
    if (total <= kFinalMaxCand) break;
  }
  if (total > kFinalMaxCand) {  // more exact ties than shared memory holds
    if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
    return;
  }
  for_each([&](uint32_t o, uint32_t j) {
    if (plen == 0 || (o >> (32 - plen)) >= prefix) {
      const int pos = atomicAdd(&n_keys, 1);
      if (pos < kFinalMaxCand) keys[pos] = (static_cast<uint64_t>(o) << 32) | static_cast<uint64_t>(~j);
    }
  });
  __syncthreads();
  const int n = n_keys;
  if (n > kFinalMaxCand || n < topk) {
    if (tid == 0) atomicOr(ctl.error, kDevErrWorkspace);
    return;
  }
  // bitonic sort, descending, over the next power of two (padding keys rank last)
  int m = 1;
  while (m < n) m <<= 1;
  for (int i = n + tid; i < m; i += kFinalThreads) keys[i] = 0ull;
  __syncthreads();
  for (int size = 2; size <= m; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = tid; i < (m >> 1); i += kFinalThreads) {
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
  // ReLU over the kept scores and the weighted sum of W2 rows (fp32), eight
  // rows in flight per thread
  float* orow = out + static_cast<size_t>(row) * d_model;
  for (int c0 = tid * 4; c0 < d_model; c0 += kFinalThreads * 4) {
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    int t = 0;
    for (; t + 8 <= topk; t += 8) {
      uint2 raw[8];
      float w[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const uint64_t key = keys[t + u];
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
      const uint64_t key = keys[t];
      const float w = fmaxf(key_score(key), 0.0f);
      const uint2 raw = __ldg(reinterpret_cast<const uint2*>(W2 + static_cast<size_t>(key_index(key)) * d_model + c0));
      a0 = fmaf(w, __uint_as_float(raw.x << 16), a0);
      a1 = fmaf(w, __uint_as_float(raw.x & 0xFFFF0000u), a1);
      a2 = fmaf(w, __uint_as_float(raw.y << 16), a2);
      a3 = fmaf(w, __uint_as_float(raw.y & 0xFFFF0000u), a3);
    }
    *reinterpret_cast<float4*>(orow + c0) = make_float4(a0, a1, a2, a3);
  }
  if (idx || score) {
    for (int t = tid; t < topk; t += kFinalThreads) {
      const uint64_t key = keys[t];
      if (idx) idx[static_cast<size_t>(row) * topk + t] = static_cast<int32_t>(key_index(key));
      if (score) score[static_cast<size_t>(row) * topk + t] = key_score(key);
    }
  }
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
  CUtensorMap tmx, tmw;
  if (!make_tmap_bf16_2d(&tmx, a.x, a.d_model, a.N, BM)) return -1;
  if (!make_tmap_bf16_2d(&tmw, a.W1, a.d_model, a.d_ff, NT)) return -1;
  if (cudaMemsetAsync(tau, 0, static_cast<size_t>(a.N) * sizeof(uint32_t), st) != cudaSuccess) return -1;
  // counts start at -1 ("not written"): the finalize reads no list whose count the first kernel did not set
  if (cudaMemsetAsync(cnt, 0xFF, static_cast<size_t>(a.N) * p.n_sl * sizeof(int), st) != cudaSuccess) return -1;
  if (cudaFuncSetAttribute(ffn_score_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(SMEM_A)) != cudaSuccess)
    return -1;
  const int grid = p.n_units < num_sms ? p.n_units : num_sms;
  ffn_score_select_kernel<<<grid, kThreads, SMEM_A, st>>>(tmx, tmw, a.N, a.d_model, a.d_ff, a.topk, p.n_rt, p.n_sl,
                                                           p.tiles, p.n_units, p.cap, cand, cnt, tau, ctl);
  if (cudaGetLastError() != cudaSuccess) return -1;
  constexpr size_t kFinalSmem = kFinalMaxCand * sizeof(uint64_t);
  if (cudaFuncSetAttribute(ffn_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kFinalSmem)) != cudaSuccess)
    return -1;
  ffn_finalize_kernel<<<a.N, kFinalThreads, kFinalSmem, st>>>(static_cast<const __nv_bfloat16*>(a.W2), a.out, a.d_model,
                                                      a.topk, p.n_sl, p.cap, cand, cnt, tau, a.idx, a.score, ctl);
  if (cudaGetLastError() != cudaSuccess) return -1;
  return 2;
}

}  // namespace topk
