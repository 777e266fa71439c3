// attn_plain.cu -- plain attention (Eq. 1, under Eq. 2's causal mask and
// per-batch key counts): the comparison path that the paper measures top-k
// attention against (Sec. 3).  Every valid key takes part in the softmax.
//
// The paper's chunked version materialises a [C, L_K] score chunk, applies
// the softmax and multiplies by V.  Here the score tile never leaves TMEM and
// registers: per 128-query tile and 128-key tile,
//   S = Q K^T          tcgen05.mma into one of two TMEM score buffers;
//   P = exp(S - m)     four softmax warps, one query row per thread, written
//                      as bf16 into one of two shared-memory buffers in the
//                      layout the next MMA reads (128-byte swizzled, K-major);
//   O += P V           tcgen05.mma into a TMEM accumulator of d columns, with
//                      V read as its transpose V^T [d, L_K] (made once per call
//                      by a transpose kernel) so that both MMAs take K-major
//                      operands.
// The running maximum m of a row is raised only when a tile's maximum exceeds
// it by more than kRescale: exp(s - m) then stays below e^kRescale, and O and
// the running sum z are scaled by exp(m_old - m_new) when it moves.  The row
// is normalised by z once, after the last key tile.
#include <cuda_bf16.h>

#include "kernels.h"

namespace topk {

namespace {

constexpr int BM = 128;           // queries per tile (TMEM lanes)
constexpr int BN = 128;           // keys per tile
constexpr float kRescale = 8.0f;  // natural-log units

template <int D>
struct PlainLayout {
  static constexpr int R = D / 64;  // 128-byte column blocks of a Q or K row
  static constexpr int S = D == 64 ? 3 : 2;
  static constexpr uint32_t Q_BYTES = BM * D * 2;
  static constexpr uint32_t K_BYTES = BN * D * 2;  // a key tile, keys x d
  static constexpr uint32_t V_BYTES = D * BN * 2;  // the same keys of V^T, d x keys (two 64-key blocks)
  static constexpr uint32_t P_BYTES = BM * BN * 2;  // one of two P buffers
  static constexpr size_t OFF_Q = 0;
  static constexpr size_t OFF_K = OFF_Q + Q_BYTES;
  static constexpr size_t OFF_V = OFF_K + static_cast<size_t>(S) * K_BYTES;
  static constexpr size_t OFF_P = OFF_V + static_cast<size_t>(S) * V_BYTES;
  static constexpr size_t OFF_BAR = OFF_P + 2 * static_cast<size_t>(P_BYTES);
  // full/empty per K/V stage, q full/empty, s full/empty per score buffer,
  // p_full/pv_done per P buffer, o_empty, drain
  static constexpr int NBARS = 2 * S + 2 + 4 + 4 + 2;
  static constexpr size_t BYTES = 1024 + OFF_BAR + NBARS * 8 + 16;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t O_COL = 2 * BN;  // O after the two score buffers
  static_assert(O_COL + D <= TMEM_COLS, "TMEM columns");
  static_assert(BYTES <= 232448, "shared memory");
};

__device__ __forceinline__ bool warp_wait_p(uint64_t* bar, uint32_t parity, const DevCtl& ctl,
                                            volatile int* abort_flag) {
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ctl, abort_flag) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  return ok != 0;
}

__device__ __forceinline__ void mbar_drain_p(uint64_t* bar, uint32_t parity, const DevCtl& ctl) {
  const unsigned long long t0 = global_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_ns() - t0 > ctl.wait_limit_ns) {
      atomicOr(ctl.error, kDevErrTimeout);
      return;
    }
  }
}

// 32 consecutive 32-bit TMEM columns of lane (taddr lane field) + thread, written.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

constexpr float kLog2e = 1.4426950408889634f;  // log2(e)

// 2^x by the hardware approximation (ex2.approx); 2^-inf = 0
__device__ __forceinline__ float ex2_approx(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

template <int D>
__global__ void __launch_bounds__(192, 1)
    attn_plain_kernel(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmk,
                      const __grid_constant__ CUtensorMap tmv, __nv_bfloat16* __restrict__ out, int BH, int H,
                      int Lq, int Lk, int causal, const int32_t* __restrict__ kv_len, int n_units, DevCtl ctl) {
  using L = PlainLayout<D>;
  constexpr int S = L::S, R = L::R;
  constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
  constexpr uint32_t IDESC_O = idesc_bf16_f32(BM, D);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* q_s = smem + L::OFF_Q;
  uint8_t* k_s = smem + L::OFF_K;
  uint8_t* v_s = smem + L::OFF_V;
  uint8_t* p_s = smem + L::OFF_P;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* full_kv = bars;
  uint64_t* empty_kv = bars + S;
  uint64_t* q_full = bars + 2 * S;
  uint64_t* q_empty = bars + 2 * S + 1;
  uint64_t* s_full = bars + 2 * S + 2;   // [2]
  uint64_t* s_empty = bars + 2 * S + 4;  // [2]
  uint64_t* p_full = bars + 2 * S + 6;   // [2]
  uint64_t* pv_done = bars + 2 * S + 8;  // [2]
  uint64_t* o_empty = bars + 2 * S + 10;
  uint64_t* drain = bars + 2 * S + 11;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + L::NBARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_kv[s], 1);
      mbar_init(&empty_kv[s], 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_empty[b], 4);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&p_full[b], 4);
      mbar_init(&pv_done[b], 1);
    }
    mbar_init(o_empty, 4);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, L::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_qt = (Lq + BM - 1) / BM;
  const int coff = Lk - Lq;
  auto decode = [&](int u, int& bh, int& qt) {
    if (causal) {  // heaviest query tiles first
      qt = n_qt - 1 - u / BH;
      bh = u % BH;
    } else {
      bh = u / n_qt;
      qt = u % n_qt;
    }
  };
  auto kv_end = [&](int bh) { return kv_len ? min(max(__ldg(kv_len + bh / H), 0), Lk) : Lk; };
  auto key_tiles = [&](int bh, int qt) {  // at least one (fully masked if the rows have no key)
    int kend = min(kv_end(bh), causal ? (qt + 1) * BM + coff : Lk);
    kend = max(kend, 1);
    return (kend + BN - 1) / BN;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmq);
      tma_prefetch_desc(&tmk);
      tma_prefetch_desc(&tmv);
    }
    uint32_t it = 0, q_issued = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int bh, qt;
      decode(u, bh, qt);
      if (!warp_wait_p(q_empty, (q_issued & 1u) ^ 1u, ctl, abort_flag)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(q_full, L::Q_BYTES);
        for (int r = 0; r < R; ++r) tma_load_3d(q_s + r * BM * 128, &tmq, q_full, r * 64, qt * BM, bh);
      }
      ++q_issued;
      const int nk = key_tiles(bh, qt);
      for (int kt = 0; kt < nk; ++kt, ++it) {
        const int s = it % S;
        if (!warp_wait_p(&empty_kv[s], ((it / S) & 1u) ^ 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&full_kv[s], L::K_BYTES + L::V_BYTES);
          uint8_t* ks = k_s + static_cast<size_t>(s) * L::K_BYTES;
          uint8_t* vs = v_s + static_cast<size_t>(s) * L::V_BYTES;
          for (int r = 0; r < R; ++r) tma_load_3d(ks + r * BN * 128, &tmk, &full_kv[s], r * 64, kt * BN, bh);
          for (int r = 0; r < 2; ++r) tma_load_3d(vs + r * D * 128, &tmv, &full_kv[s], kt * BN + r * 64, 0, bh);
        }
      }
    }
    __syncwarp();
    if (lane == 0) {  // every issued copy must land before the CTA exits
      for (uint32_t back = 1; back <= static_cast<uint32_t>(S) && back <= it; ++back) {
        const uint32_t t = it - back;
        mbar_drain_p(&full_kv[t % S], (t / S) & 1u, ctl);
      }
      if (q_issued > 0) mbar_drain_p(q_full, (q_issued - 1) & 1u, ctl);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    uint32_t it = 0, sc = 0, pc = 0, qi = 0;
    bool ok = true;
    auto issue_pv = [&](uint32_t stage, uint32_t pb, bool first) {
      const uint32_t o_tmem = tmem_base + L::O_COL;
      const uint32_t pa = smem_u32(p_s + static_cast<size_t>(pb) * L::P_BYTES);
      const uint32_t va = smem_u32(v_s + static_cast<size_t>(stage) * L::V_BYTES);
#pragma unroll
      for (int st = 0; st < BN / 16; ++st) {
        const uint32_t r = st / 4, off = (st % 4) * 32;
        mma_bf16_ss(o_tmem, sdesc_k128(pa + r * BM * 128 + off), sdesc_k128(va + r * D * 128 + off), IDESC_O,
                    (first && st == 0) ? 0u : 1u);
      }
      mma_commit(&pv_done[pb]);
      mma_commit(&empty_kv[stage]);
    };
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x, ++qi) {
      int bh, qt;
      decode(u, bh, qt);
      if (!warp_wait_p(q_full, qi & 1u, ctl, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int nk = key_tiles(bh, qt);
      uint32_t prev_stage = 0;
      for (int kt = 0; kt <= nk && ok; ++kt) {
        if (kt < nk) {
          const int s = it % S;
          const int b = sc & 1u;
          if (!warp_wait_p(&full_kv[s], (it / S) & 1u, ctl, abort_flag) ||
              !warp_wait_p(&s_empty[b], ((sc >> 1) & 1u) ^ 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) {
            const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(b * BN);
            const uint32_t qa = smem_u32(q_s);
            const uint32_t ka = smem_u32(k_s + static_cast<size_t>(s) * L::K_BYTES);
#pragma unroll
            for (int st = 0; st < D / 16; ++st) {
              const uint32_t r = st / 4, off = (st % 4) * 32;
              mma_bf16_ss(d_tmem, sdesc_k128(qa + r * BM * 128 + off), sdesc_k128(ka + r * BN * 128 + off),
                          IDESC_S, st > 0 ? 1u : 0u);
            }
            mma_commit(&s_full[b]);
          }
          __syncwarp();
        }
        if (kt > 0) {  // P of the previous key tile is ready: O += P V
          if (kt == 1 && qi > 0 && !warp_wait_p(o_empty, (qi - 1) & 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          // P number pc sits in buffer pc & 1, that buffer's (pc >> 1)-th use
          if (!warp_wait_p(&p_full[pc & 1u], (pc >> 1) & 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) issue_pv(prev_stage, pc & 1u, kt == 1);
          __syncwarp();
          ++pc;
        }
        if (kt < nk) {
          prev_stage = it % S;
          ++it;
          ++sc;
        }
      }
      if (!ok) break;
      if (lane == 0) mma_commit(q_empty);
      __syncwarp();
    }
    if (lane == 0) {  // all issued MMAs must complete before TMEM is freed
      mma_commit(drain);
      mbar_drain_p(drain, 0, ctl);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t o_taddr = tmem_base + lane_base + L::O_COL;
    uint32_t sc = 0, pc = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      int bh, qt;
      decode(u, bh, qt);
      const int i_row = qt * BM + row;
      const int nk = key_tiles(bh, qt);
      const int lim = min(kv_end(bh), causal ? min(i_row + 1 + coff, Lk) : Lk);  // keys j < lim are valid
      const int lim_min = min(kv_end(bh), causal ? min(qt * BM + 1 + coff, Lk) : Lk);  // smallest in the tile
      float m_run = -INFINITY, z = 0.f;
      for (int kt = 0; kt < nk; ++kt, ++sc) {
        const int b = sc & 1u;
        if (!warp_wait_p(&s_full[b], (sc >> 1) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float s[BN];
        const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(b * BN);
        tmem_ld64(taddr, *reinterpret_cast<float(*)[64]>(s));
        tmem_ld64(taddr + 64, *reinterpret_cast<float(*)[64]>(s + 64));
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_empty[b]);
        const int j0 = kt * BN;
        if (j0 + BN > lim_min) {  // only tiles that reach past some row's limit need the mask
#pragma unroll
          for (int e = 0; e < BN; ++e)
            if (j0 + e >= lim) s[e] = -INFINITY;
        }
        float mt = s[0];
#pragma unroll
        for (int e = 1; e + 1 < BN; e += 2) mt = max3f(mt, s[e], s[e + 1]);
        mt = fmaxf(mt, s[BN - 1]);
        const bool raise = mt > m_run + kRescale || (m_run == -INFINITY && mt > -INFINITY);
        const float m_new = raise ? mt : m_run;
        const float alpha = (raise && m_run > -INFINITY) ? ex2_approx((m_run - m_new) * kLog2e) : 1.f;
        m_run = m_new;
        // P row as packed bf16, computed before any wait on the previous products:
        // exp(s - m) = 2^(s log2(e) - m log2(e)); a row with no valid key so far has p = 0
        uint32_t w[BN / 2];
        float zp[4] = {0.f, 0.f, 0.f, 0.f};  // four partial sums: no long dependent chain
        if (m_run == -INFINITY) {
#pragma unroll
          for (int e = 0; e < BN / 2; ++e) w[e] = 0u;
        } else {
          const float ml = m_run * kLog2e;
#pragma unroll
          for (int e = 0; e < BN / 2; ++e) {
            const float p0 = ex2_approx(fmaf(s[2 * e], kLog2e, -ml));
            const float p1 = ex2_approx(fmaf(s[2 * e + 1], kLog2e, -ml));
            w[e] = pack_bf16x2(p0, p1);
            zp[e & 3] += p0 + p1;
          }
        }
        const float zt = (zp[0] + zp[1]) + (zp[2] + zp[3]);
        z = z * alpha + zt;
        // P number pc goes to buffer pc & 1, whose previous P (number pc - 2) its product must have read;
        // a rescale of O needs the previous product (number pc - 1) done as well
        const uint32_t pb = pc & 1u;
        if (pc >= 2 && !warp_wait_p(&pv_done[pb], ((pc - 2) >> 1) & 1u, ctl, abort_flag)) {
          ok = false;
          break;
        }
        if (kt > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
          if (!warp_wait_p(&pv_done[(pc - 1) & 1u], ((pc - 1) >> 1) & 1u, ctl, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < D; c += 32) {
            float o[32];
            tmem_ld32(o_taddr + c, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= alpha;
            tmem_st32(o_taddr + c, o);
          }
          tmem_wait_st();
        }
        // 128-byte swizzled K-major: row `row` of block r holds keys 64r .. 64r + 63, its 16-byte
        // chunk c at chunk position c ^ (row & 7)
        uint8_t* pbuf = p_s + static_cast<size_t>(pb) * L::P_BYTES;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          uint8_t* prow = pbuf + r * BM * 128 + row * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const int e = r * 32 + c * 4;
            *reinterpret_cast<uint4*>(prow + ((c ^ (row & 7)) << 4)) = make_uint4(w[e], w[e + 1], w[e + 2], w[e + 3]);
          }
        }
        fence_async_smem();  // the MMA (async proxy) reads what these generic stores wrote
        tc_fence_before();   // and the rescaled O above
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[pb]);
        ++pc;
      }
      if (!ok) break;
      // the last tile's P V (number pc - 1; products complete in issue order), then out = O / z
      if (!warp_wait_p(&pv_done[(pc - 1) & 1u], ((pc - 1) >> 1) & 1u, ctl, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv = z > 0.f ? 1.f / z : 0.f;
#pragma unroll 1
      for (int c = 0; c < D; c += 32) {
        float o[32];
        tmem_ld32(o_taddr + c, o);
        tmem_wait_ld();
        if (i_row < Lq) {
          uint4* dst = reinterpret_cast<uint4*>(out + (static_cast<size_t>(bh) * Lq + i_row) * D + c);
#pragma unroll
          for (int g = 0; g < 4; ++g)
            dst[g] = make_uint4(pack_bf16x2(o[8 * g] * inv, o[8 * g + 1] * inv),
                                pack_bf16x2(o[8 * g + 2] * inv, o[8 * g + 3] * inv),
                                pack_bf16x2(o[8 * g + 4] * inv, o[8 * g + 5] * inv),
                                pack_bf16x2(o[8 * g + 6] * inv, o[8 * g + 7] * inv));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_empty);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, L::TMEM_COLS);
  }
}

// V [BH][Lk][D] -> V^T [BH][D][Lkp], keys Lk .. Lkp - 1 zero.
template <int D>
__global__ void transpose_v_kernel(const __nv_bfloat16* __restrict__ v, __nv_bfloat16* __restrict__ vt, int Lk,
                                   int Lkp) {
  __shared__ __nv_bfloat16 tile[32][33];
  const int bh = blockIdx.z;
  const int j0 = blockIdx.x * 32, c0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
  for (int yy = ty; yy < 32; yy += 8) {
    const int j = j0 + yy;
    tile[yy][tx] = j < Lk ? v[(static_cast<size_t>(bh) * Lk + j) * D + c0 + tx] : __float2bfloat16(0.f);
  }
  __syncthreads();
  for (int yy = ty; yy < 32; yy += 8) {
    const int j = j0 + tx;
    if (j < Lkp) vt[(static_cast<size_t>(bh) * D + c0 + yy) * Lkp + j] = tile[tx][yy];
  }
}

template <int D>
int launch_plain(const PlainArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  using L = PlainLayout<D>;
  const int BH = a.B * a.H;
  const int Lkp = (a.Lk + 7) / 8 * 8;
  __nv_bfloat16* vt = static_cast<__nv_bfloat16*>(a.workspace);
  dim3 tg((Lkp + 31) / 32, D / 32, BH), tb(32, 8);
  transpose_v_kernel<D><<<tg, tb, 0, st>>>(static_cast<const __nv_bfloat16*>(a.v), vt, a.Lk, Lkp);
  CUtensorMap tmq, tmk, tmv;
  if (!make_tmap_bf16_3d(&tmq, a.q, D, a.Lq, BH, BM)) return -1;
  if (!make_tmap_bf16_3d(&tmk, a.k, D, a.Lk, BH, BN)) return -1;
  if (!make_tmap_bf16_3d(&tmv, vt, Lkp, D, BH, D)) return -1;
  const int n_units = BH * ((a.Lq + BM - 1) / BM);
  auto kern = attn_plain_kernel<D>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(L::BYTES)) !=
      cudaSuccess)
    return -1;
  const int grid = n_units < num_sms ? n_units : num_sms;
  kern<<<grid, 192, L::BYTES, st>>>(tmq, tmk, tmv, static_cast<__nv_bfloat16*>(a.out), BH, a.H, a.Lq, a.Lk,
                                    a.causal, a.kv_len, n_units, ctl);
  return cudaGetLastError() == cudaSuccess ? 2 : -1;
}

}  // namespace

size_t plain_workspace_bytes(int B, int H, int Lk, int d) {
  const size_t Lkp = (static_cast<size_t>(Lk) + 7) / 8 * 8;
  return static_cast<size_t>(B) * H * d * Lkp * 2;
}

int attn_plain(const PlainArgs& a, const DevCtl& ctl, int num_sms, cudaStream_t st) {
  if (a.d == 64) return launch_plain<64>(a, ctl, num_sms, st);
  if (a.d == 128) return launch_plain<128>(a, ctl, num_sms, st);
  return 0;
}

}  // namespace topk
