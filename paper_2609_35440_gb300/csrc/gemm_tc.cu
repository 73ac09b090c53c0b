// Persistent tcgen05 GEMM for sm_103a on CTA pairs, with five epilogue modes.
//
// Two CTAs on neighbouring SMs form a cluster and compute one 256 x 256
// output tile together with tcgen05.mma.cta_group::2 (M = 256, N = 256, K =
// 16, bf16 in, fp32 accumulate).  Each CTA stages its own 128 rows of A and
// its own 128 columns of B per 128-wide reduction block (64 KB), so a
// 3-stage ring fits in shared memory next to the epilogue's staging buffers,
// and each SM needs 64 B of operands per clock at full MMA rate (a single-CTA
// 128 x 256 tile needs 96 B).  Roles, in both CTAs:
//   warp 0     TMA producer: loads its CTA's A and B halves, completion is
//              signalled on the even CTA's "full" barrier (pair-mode TMA)
//   warp 1     even CTA: one thread issues the pair MMAs into one of two TMEM
//              accumulators of 256 columns and commits (multicast) to both
//              CTAs' "empty" and "tmem full" barriers; both CTAs' warp 1
//              allocate / free the tensor memory together
//   warps 2-5  epilogue: each owns 32 TMEM lanes (rows) of its CTA's 128
//              rows x 256 columns; releases the accumulator on the even CTA's
//              "tmem empty" barrier (8 arrivals: 4 warps x 2 CTAs)
//
// Work units: the pairs take units round robin.  A unit is a whole tile, or,
// for the tiles that do not fill a last complete wave of pairs (kDxhat, kDW),
// one of up to 8 contiguous ranges of the tile's reduction; part 0 of such a
// tile is stored to the output and the other parts to auxiliary slots that
// launch_split_fixup adds back in a fixed order.
//
// Epilogues:
//  kLogits  Z = Xhat W^T.  Per row and 256-column tile: m = max_v z,
//           s = sum_v exp(z - m), sum_v exp(z - m) z, the target logit when
//           the target falls in the tile, and the bf16 values exp(z - m)
//           written to a [rows, V] buffer with TMA stores.  These feed the
//           log-sum-exp of the cross-entropy (Eq. 2 and the local loss of
//           Algorithm 1), the RMSNorm backward's row sum and, rescaled, the
//           gradient, so the logits are never written and never recomputed.
//  kDxhat   dXhat = G W, the readout factor W^T delta_k of Eq. 3, and in the
//           same epilogue the final RMSNorm's backward: bf16 dH and the final
//           module's dgamma partial sums (fp32 dXhat for the cut tiles).
//  kDW      dW = G^T Xhat over the final module's tokens; fp32 out.
//  kLogitsHeads  as kLogits with each head's temperature and bias (Algorithm
//           1: z = tau_k W-bar xhat + b_k), plus per tile sum exp(z - m) s and
//           the target's s, for the temperature's gradient.
//  kExit    Z = Xhat W^T for the early exits (every depth decodes through the
//           shared readout, paper Section 3 and Appendix E): per row and tile
//           the max, the sum of exp(z - max) (online, one TMEM pass), the
//           first column reaching the max and the target logit.
//
// Every wait is bounded (ptx.cuh); on a timeout all roles unwind, in-flight
// copies and MMAs are drained, TMEM is freed and SOLO_FLAG_TIMEOUT is set.
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

#include "../../include/solo_readout.h"

namespace solo {
namespace {

constexpr int kPairRows = 2 * kBM;                  // 256 output rows per CTA pair
constexpr int kBHalf = kBN / 2;                     // B columns staged per CTA
constexpr int kABytes = kBM * kBK * 2;              // 32 KB at kBK = 128
constexpr int kBBytes = kBHalf * kBK * 2;           // 32 KB at kBK = 128
constexpr int kMnBlock = 64 * kBK * 2;              // MN-major: one 64-wide MN block
constexpr int kStageBytes = kABytes + kBBytes;      // per CTA
constexpr int kEpiBufBytes = 32 * 128;              // 32 rows x 128 B
constexpr int kEpiWarps = 4;
constexpr int kTmemCols = 2 * kBN;                  // two accumulators
constexpr int kSmemA = 0;
constexpr int kSmemB = kStages * kABytes;
constexpr int kSmemEpi = kSmemB + kStages * kBBytes;
constexpr int kSmemBar = kSmemEpi + kEpiWarps * 2 * kEpiBufBytes;
constexpr int kNumBars = 2 * kStages + 2 + 2 + 1;
constexpr int kSmemMisc = kSmemBar + kNumBars * 8;
constexpr int kSmemTotal = kSmemMisc + 16 + 1024;   // + alignment slack
static_assert(kSmemTotal <= 232448, "shared memory budget");

constexpr float kLog2e = 1.4426950408889634f;
// Exponentials are stored against the reference 0 while the tile's maximum logit
// stays within this bound (e^64 leaves fp32 and bf16 room for 2^23 terms).
constexpr float kRefBound = 64.f;

constexpr uint16_t kBothCtas = 0x3;

// The product's rows and its work units.  From the host's GemmArgs, or, with
// compacted rows (m_dev), planned here from the device row count with the
// host's rule (plan_units): whole tiles fill complete waves of pairs, the rest
// is cut along the reduction.
struct Plan {
  int M, m_blocks, num_tiles, full_tiles, split, num_units, k_blocks;
};

__device__ __forceinline__ Plan make_plan(const GemmArgs& a) {
  Plan p{a.M, a.m_blocks, a.num_tiles, a.full_tiles, a.split, a.num_units, a.k_blocks};
  if (a.m_dev == nullptr && a.kend_dev == nullptr) return p;
  if (a.m_dev != nullptr) {
    p.M = min(*a.m_dev, a.M);
    p.m_blocks = (p.M + 2 * kBM - 1) / (2 * kBM);
  }
  if (a.kend_dev != nullptr && a.row0_dev != nullptr) {
    // kDW over the final module's kept tokens (all masked: the host's length
    // over zeroed rows)
    const int rows = *a.kend_dev - *a.row0_dev;
    if (rows > 0) p.k_blocks = min((rows + kBK - 1) / kBK, a.k_blocks);
  }
  p.num_tiles = p.m_blocks * a.n_blocks;
  p.full_tiles = p.num_tiles;
  p.split = 1;
  p.num_units = p.num_tiles;
  const int pairs = min(max(a.sms / 2, 1), kMaxAuxSlots + 1);
  const int rem = p.num_tiles % pairs;
  if (!a.split_ok || rem == 0) return p;
  int s = min(min(pairs / rem, kMaxSplit), p.k_blocks);
  while (s > 1 && rem * (a.aux_part0 ? s : s - 1) > min(a.aux_slots, kMaxAuxSlots)) --s;
  if (s < 2) return p;
  p.full_tiles = p.num_tiles - rem;
  p.split = s;
  p.num_units = p.full_tiles + rem * s;
  return p;
}

__device__ __forceinline__ void tile_coords(int t, const GemmArgs& a, const Plan& p, int& mb,
                                            int& nb) {
  const int per_group = a.group_m * a.n_blocks;
  const int g = t / per_group;
  const int first_m = g * a.group_m;
  const int gm = min(p.m_blocks - first_m, a.group_m);
  const int r = t - g * per_group;
  mb = first_m + r % gm;
  nb = r / gm;
}

// Work unit u -> tile, part of the tile (0 for a whole tile) and its
// reduction blocks [kb_lo, kb_hi).
__device__ __forceinline__ void unit_range(int u, const GemmArgs& a, const Plan& p, int& t,
                                           int& part, int& kb_lo, int& kb_hi) {
  if (u < p.full_tiles) {
    t = u;
    part = 0;
    kb_lo = 0;
    kb_hi = p.k_blocks;
    return;
  }
  const int i = u - p.full_tiles;
  t = p.full_tiles + i / p.split;
  part = i % p.split;
  kb_lo = static_cast<int>(static_cast<int64_t>(part) * p.k_blocks / p.split);
  kb_hi = static_cast<int>(static_cast<int64_t>(part + 1) * p.k_blocks / p.split);
}

// Waits without looking at the abort flag, bounded in time: used to drain
// copies and MMAs that were already issued when a role gave up.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_cluster(a, parity)) {
    if (globaltimer_ns() - t0 > kWaitLimitNs) break;
  }
}

// Waits on a barrier whose phases complete by TMA transactions (the "full"
// barriers, whose bytes may come from the peer CTA's loads) or by MMA commits
// ("empty", "tmem full"): a CTA-scope acquire suffices (measured 0.7-1.2 %
// faster than a cluster-scope one).  The "tmem empty" barrier, which takes
// software arrivals from the peer CTA, is waited on at cluster scope.
__device__ __forceinline__ bool mbar_wait_hw(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return mbar_wait(bar, parity, abort);
}

// ---- the RMSNorm backward, fused into the dX̂ epilogue -----------------------
// Eq. 3 sends delta_k back through the final RMSNorm.  With dxhat = G W,
//   dh_j = r gamma_j dxhat_j - (r^3 / d) h_j S,   S = sum_l gamma_l h_l dxhat_l.
// S needs a whole row of dxhat, which one 256-column tile does not hold.  But
// gamma_l h_l r is xhat_l before its bf16 rounding, so
//   S = (1/r) sum_l xhat_l dxhat_l = (1/r) sum_v G_v s_v
//     = tau inv_nvalid (E_p[s] - s_y) / r
// (s = W xhat, the logits before temperature and bias), which the logits
// epilogue and the log-sum-exp pass reduce per row (edz).  The two forms
// differ only by xhat's rounding, far inside the gradient tolerances.

struct NormRow {
  bool ok;             // a row of the product
  bool dg;             // a row of the final module (its dgamma terms are summed)
  float r, coef;       // r_i and (r_i^3 / d) S_i
  const uint16_t* h;   // the row of hidden (bf16)
  uint16_t* dh;        // the row of dhidden (bf16)
  // dxhat = fa acc - fb W_y: the accumulator holds the stored exponentials times
  // W (a row left out of the gradient pass) or G W (fa = 1, fb = 0)
  float fa, fb;
  const uint16_t* wy;  // the row W_y, or null (fb = 0)
};

// dg_row0: first row of the final module (compacted rows: its first kept token).
__device__ __forceinline__ NormRow norm_row(const GemmArgs& g, int64_t row, int M,
                                            int64_t dg_row0) {
  NormRow nr{false, false, 0.f, 0.f, nullptr, nullptr, 1.f, 0.f, nullptr};
  if (row >= M) return nr;
  const int64_t tok = g.orig_row ? g.orig_row[row] : row;
  const int k = static_cast<int>(tok / g.tokens_per_module);
  if (!in_bounds(k < g.modules, g.flags)) return nr;
  const int64_t n = tok - static_cast<int64_t>(k) * g.tokens_per_module;
  const float r = g.r[row];
  const float tau = g.tau ? g.tau[k] : 1.f;
  nr.ok = true;
  nr.dg = g.dg_part != nullptr && row >= dg_row0;
  nr.r = r;
  nr.coef = r * r * (tau * g.inv_nvalid[k] * g.edz[row]) / static_cast<float>(g.N);
  nr.h = g.hidden[k] + n * g.N;
  nr.dh = g.dhidden[k] + n * g.N;
  if (g.row_fa != nullptr) {
    const float fa = g.row_fa[row];
    if (fa >= 0.f) {              // a row whose gradient is formed here
      const float scale = tau * g.inv_nvalid[k];
      nr.fa = scale * fa;
      nr.fb = scale * g.row_fb[row];
      const int y = g.targets[row];
      if (nr.fb != 0.f && in_bounds(y >= 0 && y < g.Vw, g.flags))
        nr.wy = g.W + static_cast<int64_t>(y) * g.N;
      else
        nr.fb = 0.f;
    }
  }
  return nr;
}

// Sum over the warp's lanes of p[j], for every j at once: after five halving
// exchanges lane j holds the sum of p[j] (31 shuffles, fixed order).
__device__ __forceinline__ float reduce_scatter32(float (&p)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 0; s < 5; ++s) {
    const int o = 16 >> s;                   // partner distance = values kept
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (i < o) {
        const float send = upper ? p[i] : p[i + o];
        const float keep = upper ? p[i + o] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
  }
  return p[0];
}

// Columns [col0, col0 + 32) of this lane's row, cols of them valid (a multiple
// of 8), dxhat in v: dH in bf16, and, when the warp holds rows of the final
// module (dg_warp, warp-uniform), the column sums over its 32 rows of
// dxhat h r, lane j storing column col0 + j at dg_dst[j].
__device__ __forceinline__ void norm_bwd_chunk(const GemmArgs& g, float (&v)[32], int col0,
                                               int cols, const NormRow& nr, bool dg_warp,
                                               float* dg_dst) {
  const int lane = threadIdx.x & 31;
  if (nr.fa != 1.f || nr.wy != nullptr) {
    // dxhat = fa acc - fb W_y
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4 wv = make_uint4(0, 0, 0, 0);
      if (nr.wy != nullptr && 8 * q < cols) wv = __ldg(reinterpret_cast<const uint4*>(nr.wy + col0) + q);
      const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = 8 * q + 2 * j;
        v[c] = fmaf(nr.fa, v[c], -nr.fb * __uint_as_float(ww[j] << 16));
        v[c + 1] = fmaf(nr.fa, v[c + 1], -nr.fb * __uint_as_float(ww[j] & 0xFFFF0000u));
      }
    }
  }
  float h[32], gm[32];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 hv = make_uint4(0, 0, 0, 0), gv = make_uint4(0, 0, 0, 0);
    if (8 * q < cols) {
      gv = __ldg(reinterpret_cast<const uint4*>(g.gamma + col0) + q);
      if (nr.ok) hv = __ldg(reinterpret_cast<const uint4*>(nr.h + col0) + q);
    }
    const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w}, gw[4] = {gv.x, gv.y, gv.z, gv.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      h[8 * q + 2 * j] = __uint_as_float(hw[j] << 16);
      h[8 * q + 2 * j + 1] = __uint_as_float(hw[j] & 0xFFFF0000u);
      gm[8 * q + 2 * j] = __uint_as_float(gw[j] << 16);
      gm[8 * q + 2 * j + 1] = __uint_as_float(gw[j] & 0xFFFF0000u);
    }
  }
  if (nr.ok) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (8 * q < cols) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int c = 8 * q + 2 * j;
          w[j] = pack_bf16x2(fmaf(nr.r * gm[c], v[c], -nr.coef * h[c]),
                             fmaf(nr.r * gm[c + 1], v[c + 1], -nr.coef * h[c + 1]));
        }
        reinterpret_cast<uint4*>(nr.dh + col0)[q] = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
  if (dg_warp) {
    float p[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) p[j] = nr.dg ? v[j] * h[j] * nr.r : 0.f;
    const float sum = reduce_scatter32(p);
    if (dg_dst != nullptr && lane < cols) dg_dst[lane] = sum;
  }
}

// The dgamma partial row of the 32-row block starting at row_base (a multiple
// of 32), for columns from col0.  Callers ask only for blocks holding a row of
// the final module; a checked build tests that and returns null otherwise.
__device__ __forceinline__ float* dg_block(const GemmArgs& g, int64_t row_base, int col0,
                                           int64_t dg_row0) {
  const int64_t rb = (row_base >> 5) - (dg_row0 >> 5);
  if (g.dg_part == nullptr || !in_bounds(rb >= 0 && rb < g.dg_blocks, g.flags)) return nullptr;
  return g.dg_part + rb * g.N + col0;
}

__device__ __forceinline__ void spin_ns(uint64_t ns) {
  const uint64_t t0 = globaltimer_ns();
  while (globaltimer_ns() - t0 < ns) __nanosleep(1000);
}

template <int MODE>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmD, const __grid_constant__ CUtensorMap tmX,
                const GemmArgs args) {
  constexpr bool kAmn = (MODE == kDW);
  constexpr bool kBmn = (MODE == kDxhat || MODE == kDW);
  constexpr uint32_t kIdesc = idesc_bf16_f32(kPairRows, kBN, kAmn, kBmn);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kSmemBar);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* tfull = bars + 2 * kStages;
  uint64_t* tempty = bars + 2 * kStages + 2;
  uint64_t* drain = bars + 2 * kStages + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kSmemMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kSmemMisc + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();       // 0: even CTA (issues the MMAs), 1: odd
  const bool even = rank == 0;
  const int cluster = blockIdx.x >> 1;
  const int num_clusters = gridDim.x >> 1;
  const Plan plan = make_plan(args);
  // kDW: first reduction row (the final module's first token); kDxhat: first
  // row of the final module, for the dgamma blocks; read from device memory
  // when the rows are compacted
  const int64_t dev_row0 = args.row0_dev ? static_cast<int64_t>(*args.row0_dev) : -1;
  const int64_t kred0 = (MODE == kDW && dev_row0 >= 0) ? dev_row0 : args.k_row0;
  const int64_t row0 = (MODE == kDxhat && dev_row0 >= 0) ? dev_row0 : args.dg_row0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbarrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmD);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();            // the peer's barriers exist before anything signals them
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint32_t full_even = map_to_rank(smem_u32(full), 0);
      uint32_t stage = 0, phase = 0;
      uint32_t issued = 0, last_phase = 0;   // per-stage bits for draining
      bool ok = true;
      for (int u = cluster; ok && u < plan.num_units; u += num_clusters) {
        int t, part, kb_lo, kb_hi, mb, nb;
        unit_range(u, args, plan, t, part, kb_lo, kb_hi);
        tile_coords(t, args, plan, mb, nb);
        const int m0 = mb * kPairRows + static_cast<int>(rank) * kBM;
        const int n0 = nb * kBN + static_cast<int>(rank) * kBHalf;
        for (int kb = kb_lo; kb < kb_hi; ++kb) {
          if (!mbar_wait_hw(&empty[stage], phase ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sA = smem + kSmemA + stage * kABytes;
          uint8_t* sB = smem + kSmemB + stage * kBBytes;
          if (even) mbar_arrive_expect_tx(&full[stage], 2 * kStageBytes);
          const uint32_t fb = full_even + stage * 8;
          const int kr = static_cast<int>(kred0) + kb * kBK;
          if constexpr (!kAmn) {
#pragma unroll
            for (int a = 0; a < kKAtoms; ++a)
              tma_load_2d_pair(sA + a * kBM * 128, &tmA, fb, kb * kBK + 64 * a, m0);
          } else {
#pragma unroll
            for (int c = 0; c < kBM / 64; ++c)
              tma_load_2d_pair(sA + c * kMnBlock, &tmA, fb, m0 + 64 * c, kr);
          }
          if constexpr (!kBmn) {
#pragma unroll
            for (int a = 0; a < kKAtoms; ++a)
              tma_load_2d_pair(sB + a * kBHalf * 128, &tmB, fb, kb * kBK + 64 * a, n0);
          } else {
#pragma unroll
            for (int c = 0; c < kBHalf / 64; ++c)
              tma_load_2d_pair(sB + c * kMnBlock, &tmB, fb, n0 + 64 * c, kr);
          }
          issued |= 1u << stage;
          last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (ok) {
        // Tail: wait until the MMAs have released every stage, so that no
        // commit arrival is still pending when the CTA exits.
        for (int i = 0; ok && i < kStages; ++i) {
          ok = mbar_wait_hw(&empty[stage], phase ^ 1, abort_flag);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) {
        atomicOr(args.flags, SOLO_FLAG_TIMEOUT);
        if (even) {
          // the even CTA's full barriers count both CTAs' bytes
          for (int s = 0; s < kStages; ++s)
            if (issued & (1u << s)) mbar_drain(&full[s], (last_phase >> s) & 1u);
        } else {
          spin_ns(200000);   // let this CTA's in-flight loads land
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (even && lane == 0) {
      uint32_t stage = 0, phase = 0;
      int local = 0;
      bool ok = true;
      const uint32_t a_base = smem_u32(smem + kSmemA);
      const uint32_t b_base = smem_u32(smem + kSmemB);
      for (int u = cluster; ok && u < plan.num_units; u += num_clusters, ++local) {
        int t, part, kb_lo, kb_hi;
        unit_range(u, args, plan, t, part, kb_lo, kb_hi);
        const uint32_t acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!mbar_wait_cluster(&tempty[acc], acc_phase ^ 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * kBN;
        for (int kb = kb_lo; kb < kb_hi; ++kb) {
          if (!mbar_wait_hw(&full[stage], phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = a_base + stage * kABytes;
          const uint32_t sb = b_base + stage * kBBytes;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            // K-major: 16-wide K steps within a 64-wide swizzle atom, atoms one
            // after the other; MN-major: 16 K rows of 128 B, MN blocks kMnBlock apart
            const uint64_t ad =
                kAmn ? smem_desc_sw128(sa + k * 2048, kMnBlock, 1024)
                     : smem_desc_sw128(sa + (k / 4) * kBM * 128 + (k % 4) * 32, 16, 1024);
            const uint64_t bd =
                kBmn ? smem_desc_sw128(sb + k * 2048, kMnBlock, 1024)
                     : smem_desc_sw128(sb + (k / 4) * kBHalf * 128 + (k % 4) * 32, 16, 1024);
            mma_bf16_pair(d_tmem, ad, bd, kIdesc, (kb != kb_lo || k != 0) ? 1u : 0u);
          }
          mma_commit_pair(&empty[stage], kBothCtas);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit_pair(&tfull[acc], kBothCtas);
      }
      if (!ok) {
        atomicOr(args.flags, SOLO_FLAG_TIMEOUT);
        mma_commit_pair(drain, 0x1);
        mbar_drain(drain, 0);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;                  // TMEM lane quadrant = row block of 32
    const int ew = warp - 2;                 // staging buffer owner
    uint8_t* ebuf = smem + kSmemEpi + ew * 2 * kEpiBufBytes;
    const uint32_t tempty_even = map_to_rank(smem_u32(tempty), 0);
    int buf = 0;
    int local = 0;
    bool ok = true;
    for (int u = cluster; u < plan.num_units; u += num_clusters, ++local) {
      int t, part, kb_lo, kb_hi, mb, nb;
      unit_range(u, args, plan, t, part, kb_lo, kb_hi);
      tile_coords(t, args, plan, mb, nb);
      const int m0 = mb * kPairRows + static_cast<int>(rank) * kBM;
      const int n0 = nb * kBN;
      const uint32_t acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      ok = __all_sync(0xffffffffu, mbar_wait_hw(&tfull[acc], acc_phase, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(32 * q) << 16) + acc * kBN;
      const int row = m0 + 32 * q + lane;
      const int ncols = min(kBN, args.N - n0);    // valid columns, warp-uniform

      if constexpr (MODE == kExit) {
        const bool row_ok = row < plan.M;
        const int y = (row_ok && args.targets) ? args.targets[row] : -1;
        const int yrel = y - n0;
        const bool has_y = row_ok && y >= 0 && y < args.V && yrel >= 0 && yrel < ncols;
        float mx = -INFINITY, zyv = 0.f;
        float2 sacc = make_float2(0.f, 0.f);    // sum of exp(z - mx), even and odd columns
        int amax = 0;
        for (int c = 0; c < kBN / 32; ++c) {
          if (c * 32 >= ncols) break;
          float v[32];
          tmem_ld32(tbase + c * 32, v);
          // the target logit, in the chunks holding some lane's target only
          const int yc = has_y ? yrel - c * 32 : -1;
          if (__any_sync(0xffffffffu, static_cast<unsigned>(yc) < 32u)) {
#pragma unroll
            for (int j = 0; j < 32; ++j) zyv = (j == yc) ? v[j] : zyv;
          }
          if (c * 32 + 32 > ncols) {   // ragged last chunk (warp-uniform): columns
                                       // past N neither win the max nor add to the sum
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (c * 32 + j >= ncols) v[j] = -INFINITY;
          }
          float t[11];
#pragma unroll
          for (int i = 0; i < 10; ++i) t[i] = fmax3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
          t[10] = fmaxf(v[30], v[31]);
          const float cm = fmax3(fmax3(t[0], t[1], t[2]), fmax3(t[3], t[4], t[5]),
                                 fmax3(t[6], t[7], fmax3(t[8], t[9], t[10])));
          if (__any_sync(0xffffffffu, cm > mx)) {
            int ci = 0;                           // the first column of the chunk holding cm
#pragma unroll
            for (int j = 31; j >= 0; --j) ci = (v[j] == cm) ? j : ci;
            if (cm > mx) {                        // strict: an earlier equal maximum stays
              const float f = ex2_approx((mx - cm) * kLog2e);   // rescale to the new max
              sacc = make_float2(sacc.x * f, sacc.y * f);
              mx = cm;
              amax = c * 32 + ci;
            }
          }
          const float mlog = mx * kLog2e;
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            const float2 a =
                __ffma2_rn(make_float2(v[j], v[j + 1]), make_float2(kLog2e, kLog2e),
                           make_float2(-mlog, -mlog));
            sacc = __fadd2_rn(sacc, make_float2(ex2_approx(a.x), ex2_approx(a.y)));
          }
        }
        const float ssum = sacc.x + sacc.y;
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (even) mbar_arrive_relaxed(&tempty[acc]);
          else mbar_arrive_remote_relaxed(tempty_even + acc * 8);
        }
        if (row_ok && in_bounds(nb < args.n_blocks, args.flags)) {
          args.stats[static_cast<size_t>(nb) * args.M + row] = make_float2(mx, ssum);
          args.argmax[static_cast<size_t>(nb) * args.M + row] = n0 + amax;
        }
        if (has_y) args.zy[row] = zyv;
      } else if constexpr (MODE == kLogits || MODE == kLogitsHeads) {
        constexpr bool kHeads = (MODE == kLogitsHeads);
        const bool row_ok = row < plan.M;
        const int y = row_ok ? args.targets[row] : -1;
        const int yrel = y - n0;
        const bool has_y = row_ok && y >= 0 && y < args.V && yrel >= 0 && yrel < ncols;
        // z = tau s + b for this row's module (kHeads), z = s otherwise
        float tau = 1.f;
        const float* brow = nullptr;
        if constexpr (kHeads) {
          const int64_t tok = row_ok ? (args.orig_row ? args.orig_row[row] : row) : 0;
          const int kmod = static_cast<int>(tok / args.tokens_per_module);
          if (args.tau) tau = args.tau[kmod];
          if (args.bias &&
              in_bounds(kmod < args.M / args.tokens_per_module && n0 + ncols <= args.V,
                        args.flags))
            brow = args.bias + static_cast<size_t>(kmod) * args.V + n0;
        }
        // bias of one 32-column chunk; rows of a tile share their module, so a
        // warp's vector loads hit the same addresses
        const bool bias_vec = (args.V & 3) == 0;
        auto load_bias = [&](int c, float (&b)[32]) {
          if (brow != nullptr && bias_vec && c * 32 + 32 <= ncols) {
            // the common case: eight 16-byte loads fill every value
            const float4* b4 = reinterpret_cast<const float4*>(brow + c * 32);
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
              const float4 t = __ldg(b4 + q4);
              b[4 * q4] = t.x; b[4 * q4 + 1] = t.y; b[4 * q4 + 2] = t.z; b[4 * q4 + 3] = t.w;
            }
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              b[j] = (brow != nullptr && c * 32 + j < ncols) ? __ldg(brow + c * 32 + j) : 0.f;
          }
        };
        // One pass over the accumulator takes the tile's exponentials against the
        // reference 0 and finds its maximum on the way.  They are taken against a
        // reference shared by all the row's tiles, 0, unless the tile's maximum
        // lies beyond +-kRefBound (then the maximum itself): a row all of whose
        // tiles use 0 has a gradient that is its stored exponentials times one
        // factor per row, which the dX̂ epilogue applies; only the other rows need
        // the gradient pass.  A warp holding such a row (rare) runs the pass again
        // against the maximum once the first pass's stores have landed.
        float mx = -INFINITY, zyv = 0.f, syv = 0.f, ref = 0.f;
        // the sums of exp(z - ref) and of exp(z - ref) s, each in the two lanes of a
        // packed pair (even and odd columns)
        float2 sacc = make_float2(0.f, 0.f);
        float2 uacc = make_float2(0.f, 0.f);
        for (int pass = 0; pass < 2; ++pass) {
          const float mlog = ref * kLog2e;
          mx = -INFINITY;
          sacc = make_float2(0.f, 0.f);
          uacc = make_float2(0.f, 0.f);
          // the bias of the next chunk is loaded while this one is worked on
          float bnext[32];
          if constexpr (kHeads) load_bias(0, bnext);
          for (int cp = 0; cp < kBN / 64; ++cp) {
            if (cp * 64 >= ncols) break;
            if (lane == 0) bulk_wait_group_read<1>();
            __syncwarp();
            const uint32_t srow = smem_u32(ebuf + buf * kEpiBufBytes) + lane * 128;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
              const int c = 2 * cp + half;
              float v[32], bb[32];
              if (c * 32 < ncols) {
                tmem_ld32(tbase + c * 32, v);
#pragma unroll
                for (int j = 0; j < 32; ++j) bb[j] = kHeads ? bnext[j] : 0.f;
                if constexpr (kHeads) {
                  if ((c + 1) * 32 < ncols) load_bias(c + 1, bnext);
                }
              } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = bb[j] = 0.f;
              }
              uint32_t p[16];
              const bool ragged = c * 32 + 32 > ncols;      // warp-uniform
              float z[32];
#pragma unroll
              for (int j = 0; j < 32; j += 2) {
                float2 zz = make_float2(v[j], v[j + 1]);
                if constexpr (kHeads)
                  zz = __ffma2_rn(make_float2(tau, tau), zz, make_float2(bb[j], bb[j + 1]));
                z[j] = zz.x;
                z[j + 1] = zz.y;
              }
              // the target logit, in the chunks holding some lane's target only
              const int ycol = has_y ? yrel - c * 32 : -1;
              const bool ychunk = __any_sync(0xffffffffu, static_cast<unsigned>(ycol) < 32u);
              if (ychunk) {
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                  zyv = (j == ycol) ? z[j] : zyv;
                  if constexpr (kHeads) syv = (j == ycol) ? v[j] : syv;
                }
              }
              if (ragged) {                 // columns past N take no part in the max
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (c * 32 + j >= ncols) z[j] = -INFINITY;
              }
              // the running maximum (the target's logit included): a tree of
              // three-input maxima
              {
                float t[11];
#pragma unroll
                for (int i = 0; i < 10; ++i) t[i] = fmax3(z[3 * i], z[3 * i + 1], z[3 * i + 2]);
                t[10] = fmax3(z[30], z[31], mx);
                mx = fmax3(fmax3(t[0], t[1], t[2]), fmax3(t[3], t[4], t[5]),
                           fmax3(t[6], t[7], fmax3(t[8], t[9], t[10])));
              }
              // The target's own term is left out of the tile's sums and of the
              // stored exponentials (the gradient pass writes the target entry
              // itself): the log-sum-exp pass forms lse - z_y = log1p(sum over
              // v != y of exp(z_v - z_y)), so that 1 - p_y and E_p[s] - s_y of a
              // confident row do not cancel.
              if (ychunk) {
#pragma unroll
                for (int j = 0; j < 32; ++j) z[j] = j == ycol ? -INFINITY : z[j];
              }
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float2 a = __ffma2_rn(make_float2(z[2 * j], z[2 * j + 1]),
                                            make_float2(kLog2e, kLog2e),
                                            make_float2(-mlog, -mlog));
                float e0 = ex2_approx(a.x);
                float e1 = ex2_approx(a.y);
                if (ragged) {
                  const int col = c * 32 + 2 * j;
                  e0 = col < ncols ? e0 : 0.f;
                  e1 = col + 1 < ncols ? e1 : 0.f;
                }
                sacc = __fadd2_rn(sacc, make_float2(e0, e1));
                uacc = __ffma2_rn(make_float2(e0, e1), make_float2(v[2 * j], v[2 * j + 1]), uacc);
                p[j] = pack_bf16x2(e0, e1);
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const uint32_t chunk = static_cast<uint32_t>(half * 4 + u) ^ (lane & 7);
                st_shared_v4(srow + (chunk << 4), p[4 * u], p[4 * u + 1], p[4 * u + 2],
                             p[4 * u + 3]);
              }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmD, ebuf + buf * kEpiBufBytes, n0 + cp * 64, m0 + 32 * q);
              bulk_commit_group();
            }
            buf ^= 1;
          }
          if (pass == 1) break;
          const bool redo = fabsf(mx) > kRefBound;
          if (!__any_sync(0xffffffffu, redo)) break;
          ref = redo ? mx : 0.f;
          // the second pass overwrites the stored tiles: the first pass's stores
          // must have completed
          if (lane == 0) bulk_wait_group<0>();
          __syncwarp();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (even) mbar_arrive_relaxed(&tempty[acc]);
          else mbar_arrive_remote_relaxed(tempty_even + acc * 8);
        }
        const float ssum = sacc.x + sacc.y;
        if (row_ok && in_bounds(nb < args.n_blocks, args.flags)) {
          args.stats[static_cast<size_t>(nb) * args.M + row] = make_float2(ref, ssum);
          args.usum[static_cast<size_t>(nb) * args.M + row] = uacc.x + uacc.y;
        }
        if constexpr (kHeads) {
          if (has_y) args.sy[row] = syv;
        }
        if (has_y) args.zy[row] = zyv;
      } else if (MODE == kDxhat && args.norm_fused && t < plan.full_tiles) {
        // whole dX̂ tile: the RMSNorm backward straight from TMEM to bf16 dH
        const NormRow nr = norm_row(args, row, plan.M, row0);
        const bool dg_warp = __any_sync(0xffffffffu, nr.dg);
        float* dg = dg_warp ? dg_block(args, m0 + 32 * q, n0, row0) : nullptr;
        for (int c = 0; c < kBN / 32; ++c) {
          if (c * 32 >= ncols) break;
          float v[32];
          tmem_ld32(tbase + c * 32, v);
          norm_bwd_chunk(args, v, n0 + c * 32, min(32, ncols - c * 32), nr, dg_warp,
                         dg ? dg + c * 32 : nullptr);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (even) mbar_arrive_relaxed(&tempty[acc]);
          else mbar_arrive_remote_relaxed(tempty_even + acc * 8);
        }
      } else {
        for (int c = 0; c < kBN / 32; ++c) {
          if (c * 32 >= ncols) break;
          float v[32];
          tmem_ld32(tbase + c * 32, v);
          if (lane == 0) bulk_wait_group_read<1>();
          __syncwarp();
          const uint32_t srow = smem_u32(ebuf + buf * kEpiBufBytes) + lane * 128;
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const uint32_t chunk = static_cast<uint32_t>(u) ^ (lane & 7);
            st_shared_v4(srow + (chunk << 4), __float_as_uint(v[4 * u]),
                         __float_as_uint(v[4 * u + 1]), __float_as_uint(v[4 * u + 2]),
                         __float_as_uint(v[4 * u + 3]));
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (part == 0 && !args.aux_part0) {
              tma_store_2d(&tmD, ebuf + buf * kEpiBufBytes, n0 + c * 32, m0 + 32 * q);
            } else {    // a reduction range of a cut tile: its auxiliary slot
              const int cut = t - plan.full_tiles;
              const int slot = args.aux_part0 ? cut * plan.split + part
                                              : cut * (plan.split - 1) + part - 1;
              if (in_bounds(slot >= 0 && slot < args.aux_slots, args.flags))
                tma_store_2d(&tmX, ebuf + buf * kEpiBufBytes, c * 32,
                             slot * kPairRows + static_cast<int>(rank) * kBM + 32 * q);
            }
            bulk_commit_group();
          }
          buf ^= 1;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (even) mbar_arrive_relaxed(&tempty[acc]);
          else mbar_arrive_remote_relaxed(tempty_even + acc * 8);
        }
      }
    }
    if (!ok && lane == 0) atomicOr(args.flags, SOLO_FLAG_TIMEOUT);
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();            // no CTA leaves while its peer may still signal it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

template <int MODE>
cudaError_t set_smem_attr() {
  return cudaFuncSetAttribute(gemm_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kSmemTotal);
}

}  // namespace

size_t gemm_smem_bytes() { return kSmemTotal; }

cudaError_t gemm_prepare(int /*device*/) {
  cudaError_t e = set_smem_attr<kLogits>();
  if (e == cudaSuccess) e = set_smem_attr<kDxhat>();
  if (e == cudaSuccess) e = set_smem_attr<kDW>();
  if (e == cudaSuccess) e = set_smem_attr<kExit>();
  if (e == cudaSuccess) e = set_smem_attr<kLogitsHeads>();
  return e;
}

void plan_units(GemmArgs& g, int sms, bool allow_split) {
  g.sms = sms;
  g.split_ok = allow_split ? 1 : 0;
  g.full_tiles = g.num_tiles;
  g.split = 1;
  g.num_units = g.num_tiles;
  const int pairs = std::min(std::max(sms / 2, 1), kMaxAuxSlots + 1);
  const int rem = g.num_tiles % pairs;
  if (!allow_split || rem == 0) return;
  int s = std::min({pairs / rem, kMaxSplit, g.k_blocks});
  while (s > 1 && rem * (g.aux_part0 ? s : s - 1) > std::min(g.aux_slots, kMaxAuxSlots)) --s;
  if (s < 2) return;
  g.full_tiles = g.num_tiles - rem;
  g.split = s;
  g.num_units = g.full_tiles + rem * s;
}

namespace {

// out[tile] += aux parts 1 .. split-1 of each cut tile, in that order.
// Grid (cut tiles, 256 / 16 row chunks), 256 threads: 16 rows x 64 float4.
__global__ void __launch_bounds__(256) split_fixup_kernel(const GemmArgs g, float* out,
                                                          int64_t ld, const float* aux) {
  const Plan plan = make_plan(g);
  const int cut = blockIdx.x;
  if (cut >= plan.num_tiles - plan.full_tiles) return;
  const int t = plan.full_tiles + cut;
  int mb, nb;
  tile_coords(t, g, plan, mb, nb);
  const int lr = blockIdx.y * 16 + (threadIdx.x >> 6);     // row within the tile (+ 4 x 4)
  const int c4 = threadIdx.x & 63;                          // float4 column within the tile
  const int col = nb * kBN + 4 * c4;
  for (int rr = 0; rr < 16; rr += 4) {
    const int r = lr + rr;
    const int64_t row = static_cast<int64_t>(mb) * kPairRows + r;
    if (row >= plan.M || col >= g.N) continue;     // N is a multiple of 8: whole float4s
    float4* o = reinterpret_cast<float4*>(out + row * ld + col);
    float4 acc = *o;
    for (int p = 1; p < plan.split; ++p) {
      const int slot = cut * (plan.split - 1) + p - 1;
      if (!in_bounds(slot < g.aux_slots, g.flags)) continue;
      const float4 x = *reinterpret_cast<const float4*>(
          aux + (static_cast<int64_t>(slot) * kPairRows + r) * kBN + 4 * c4);
      acc.x += x.x;
      acc.y += x.y;
      acc.z += x.z;
      acc.w += x.w;
    }
    *o = acc;
  }
}

// kDxhat with norm_fused: the RMSNorm backward of the cut tiles, from the sum
// of their fp32 parts in the auxiliary buffer (part 0 first, then 1, 2, ...:
// the order split_fixup_kernel adds them in).  Grid (cut tiles, 8 blocks of 32
// rows); warp w handles the tile's columns [32 w, 32 w + 32), lane i row i.
__global__ void __launch_bounds__(256) cut_tiles_norm_kernel(const GemmArgs g, const float* aux) {
  const Plan plan = make_plan(g);
  const int cut = static_cast<int>(blockIdx.x);
  if (cut >= plan.num_tiles - plan.full_tiles) return;   // (launched for the most cut tiles)
  const int t = plan.full_tiles + cut;
  int mb, nb;
  tile_coords(t, g, plan, mb, nb);
  const int64_t row0 = g.row0_dev ? static_cast<int64_t>(*g.row0_dev) : g.dg_row0;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int lr = blockIdx.y * 32 + lane;                    // row within the tile
  const int64_t row_base = static_cast<int64_t>(mb) * kPairRows + blockIdx.y * 32;
  const int64_t row = row_base + lane;
  const int col0 = nb * kBN + warp * 32;
  if (col0 >= g.N) return;                       // warp-uniform
  const int cols = min(32, g.N - col0);
  const NormRow nr = norm_row(g, row, plan.M, row0);
  float v[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = 0.f;
  if (nr.ok) {
    for (int p = 0; p < plan.split; ++p) {
      const int slot = cut * plan.split + p;
      if (!in_bounds(slot < g.aux_slots, g.flags)) continue;
      const float4* src = reinterpret_cast<const float4*>(
          aux + (static_cast<int64_t>(slot) * kPairRows + lr) * kBN + warp * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (4 * q < cols) {
          const float4 x = src[q];
          if (p == 0) {
            v[4 * q] = x.x;
            v[4 * q + 1] = x.y;
            v[4 * q + 2] = x.z;
            v[4 * q + 3] = x.w;
          } else {
            v[4 * q] += x.x;
            v[4 * q + 1] += x.y;
            v[4 * q + 2] += x.z;
            v[4 * q + 3] += x.w;
          }
        }
      }
    }
  }
  const bool dg_warp = __any_sync(0xffffffffu, nr.dg);
  norm_bwd_chunk(g, v, col0, cols, nr, dg_warp,
                 dg_warp ? dg_block(g, row_base, col0, row0) : nullptr);
}

}  // namespace

cudaError_t launch_cut_tiles_norm(const GemmArgs& g, const float* aux, cudaStream_t stream) {
  // compacted rows: the device plans the cut tiles; launch for the most there can be
  const int pairs = std::min(std::max(g.sms / 2, 1), kMaxAuxSlots + 1);
  const int cut = g.m_dev ? std::min(pairs - 1, g.num_tiles) : g.num_tiles - g.full_tiles;
  if (!g.norm_fused || !g.aux_part0 || cut <= 0 || (!g.m_dev && g.split < 2)) return cudaSuccess;
  cut_tiles_norm_kernel<<<dim3(cut, kPairRows / 32), 256, 0, stream>>>(g, aux);
  return launched();
}

cudaError_t launch_split_fixup(const GemmArgs& g, float* out, int64_t ld, const float* aux,
                               cudaStream_t stream) {
  const int cut = g.num_tiles - g.full_tiles;
  if (g.split < 2 || cut <= 0) return cudaSuccess;
  split_fixup_kernel<<<dim3(cut, kPairRows / 16), 256, 0, stream>>>(g, out, ld, aux);
  return launched();
}

cudaError_t launch_gemm(GemmMode mode, const CUtensorMap& a, const CUtensorMap& b,
                        const CUtensorMap& d, const CUtensorMap& x, const GemmArgs& args,
                        int sms, cudaStream_t stream) {
  if (args.num_units <= 0) return cudaSuccess;
  const int clusters = std::min(args.num_units, std::max(sms / 2, 1));
  const int grid = 2 * clusters;
  switch (mode) {
    case kLogits:
      gemm_kernel<kLogits><<<grid, kGemmThreads, kSmemTotal, stream>>>(a, b, d, x, args);
      break;
    case kDxhat:
      gemm_kernel<kDxhat><<<grid, kGemmThreads, kSmemTotal, stream>>>(a, b, d, x, args);
      break;
    case kDW:
      gemm_kernel<kDW><<<grid, kGemmThreads, kSmemTotal, stream>>>(a, b, d, x, args);
      break;
    case kExit:
      gemm_kernel<kExit><<<grid, kGemmThreads, kSmemTotal, stream>>>(a, b, d, x, args);
      break;
    case kLogitsHeads:
      gemm_kernel<kLogitsHeads><<<grid, kGemmThreads, kSmemTotal, stream>>>(a, b, d, x, args);
      break;
  }
  return launched();
}

}  // namespace solo
