// Single-pass on-chip forward + backward of the auxiliary modules.
//
// For the K-1 auxiliary modules nothing of size tokens x vocabulary touches
// global memory.  Written out, Eq. 3's readout factor of one token is
//   dxhat = (1 / Nvalid) (sum_v p_v W_v - W_y)
//         = (1 / Nvalid) ((sum over v != y of e^{z_v - m} W_v) / S - (S' / S) W_y),
//   S' = sum over v != y of e^{z_v - m},  S = S' + e^{z_y - m},
// for any reference m, and the cross-entropy of Eq. 2 is lse - z_y with
// lse = m + ln S.  So one sweep over the vocabulary in tiles yields both: per
// tile the logits z = xhat W^T, their exponentials P = e^{z - m} (target
// column left out), and O += P W; at the end dxhat = (O / S - (S'/S) W_y) / Nvalid.
// This is the attention-forward pattern with keys = values = W.
//
// Layout on GB300: O for 128 rows needs 128 x d fp32, more than the 512 columns
// of tensor memory once d > 256, so a cluster of C CTAs (C = 1, 2, 4, 8) shares
// a block of 128 rows and CTA c owns d-columns [c ds, c ds + ds) of O.  Per
// 64-column vocabulary tile each CTA:
//   - multiplies its slice of xhat (kept in tensor memory as the A operand)
//     by its slice of the W tile: a partial Z, a split of the d-sum;
//   - sends every row of the partial Z to the CTA that owns the row's
//     statistics (rows [c R, c R + R), R = 128 / C) with st.async;
//   - as owner: adds the C partials in a fixed order, tracks the row maximum,
//     forms P = bf16(e^{z - m}) and broadcasts its rows of P to the cluster
//     with bulk copies;
//   - accumulates O += P W_slice (W tile reused from shared memory, MN-major).
// Partial Z, P and the owners' receive buffers are double-buffered and the O
// product of tile t is issued after the partial Z of tile t + 2, so the
// exchanges of two tiles are in flight while the tensor core works; the
// exchange (fp32 partials, 7/8 of 32 KB out and in per CTA and tile at C = 8,
// plus bf16 P) is what bounds the pass: distributed shared memory moves
// about 15-18 B/clk per SM on GB300 (measured), against 64 B/clk of operands
// the tensor core reads.
// The reference m of a row is the maximum of its first tile; it is not moved
// while the logits stay within 64 of it (e^64 fits fp32 and bf16 with room
// for V terms).  A row whose maximum exceeds that has its whole block swept a
// second time with m set to the exact maximum of the first sweep.
//
// Roles (320 threads): warp 0 TMA producer of the W tiles; warp 1 MMA issuer
// and tensor-memory owner; warps 2-5 "lane" warps (tensor-memory lanes: xhat
// slice in, partial Z out, O out to dH with the final RMSNorm's backward);
// warps 6-9 owners (statistics, P).  Every wait is bounded; on a timeout every
// role unwinds and SOLO_FLAG_TIMEOUT is set.
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"

#include "../../include/solo_readout.h"

namespace solo {
namespace {

constexpr int kFR = 128;                       // rows per block (tensor-memory lanes)
constexpr int kFV = 64;                        // vocabulary columns per tile
constexpr int kFDS = 256;                      // widest d-slice of one CTA
constexpr int kFThreads = 320;
constexpr int kFStages = 4;                    // W tiles in flight
constexpr int kFLag = 2;                       // tiles the O product trails the partial Z
constexpr int kFAtom = kFV * 128;              // one 64-column swizzle atom of a W tile (8 KB)
constexpr int kFStageBytes = kFV * kFDS * 2;   // a W tile slice: 32 KB
constexpr int kFPBytes = kFR * kFV * 2;        // a P tile: bf16, K-major, one atom (16 KB)
// Partial-Z rows received as owner, fp32: the 16 quads (16 B) of a row sit at
// positions quad ^ (row & 15), so that the owners' float4 reads and the senders'
// stores spread over all banks.
constexpr int kFPartBytes = kFR * kFV * 4;     // 32 KB
constexpr int kFSmemP = kFStages * kFStageBytes;
constexpr int kFSmemPart = kFSmemP + 2 * kFPBytes;
constexpr int kFSmemBar = kFSmemPart + 2 * kFPartBytes;
constexpr int kFNumBars = 2 * kFStages + 6 * 2 + 5;
constexpr int kFSmemMisc = kFSmemBar + kFNumBars * 8;
constexpr int kFSmemTotal = kFSmemMisc + 32 + 1024;   // + alignment slack
static_assert(kFSmemTotal <= 232448, "shared memory budget");
// tensor-memory columns
constexpr uint32_t kTX = 0;      // xhat slice: ds bf16 = ds / 2 columns
constexpr uint32_t kTZ = 128;    // two partial-Z buffers of 64 columns
constexpr uint32_t kTO = 256;    // O slice: ds columns
constexpr float kMoveRef = 64.f; // a logit this far above the reference forces a second sweep
constexpr float kLog2e = 1.4426950408889634f;

// Barriers ([2] = one per buffer of a double-buffered resource; buffer t & 1
// serves tile t, and its phase for tile t is (t >> 1) & 1).
enum Bar {
  bWfull = 0,                    // [kFStages] W stage loaded (TMA bytes)
  bWempty = bWfull + kFStages,   // [kFStages] W stage free (MMA commit after its O product)
  bZfull = bWempty + kFStages,   // [2] partial Z in tensor memory (MMA commit)
  bZempty = bZfull + 2,          // [2] partial Z read out (4 lane warps)
  bPfull = bZempty + 2,          // [2] P tile complete in this CTA (own rows: arrive; others: bytes)
  bPfree = bPfull + 2,           // [2] every CTA's O product of the buffer's last tile done
  bPartFull = bPfree + 2,        // [2] partial-Z rows of all C CTAs received (bytes)
  bPartFree = bPartFull + 2,     // [2] every owner consumed this CTA's partials of the buffer
  bXready = bPartFree + 2,       // sweep announced, xhat slice in tensor memory (4 lane warps)
  bOfull,                        // O of the sweep complete (MMA commit)
  bOempty,                       // O read out (4 lane warps)
  bRfull,                        // per-row factors of the sweep received (bytes)
  bDrain
};
static_assert(bDrain + 1 == kFNumBars, "barrier count");

struct SweepInfo {
  int valid;
  int rb;
  int redo;
  int pad;
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_cluster(a, parity)) {
    if (globaltimer_ns() - t0 > kWaitLimitNs) break;
  }
}

__device__ __forceinline__ bool row_kept(const FlashArgs& a, int64_t row, int y) {
  return y >= 0 && y < a.V && y != a.ignore_index && (a.mask == nullptr || a.mask[row] != 0);
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <int C>
__global__ void __cluster_dims__(C, 1, 1) __launch_bounds__(kFThreads, 1)
    flash_bwd_kernel(const __grid_constant__ CUtensorMap tmW, const FlashArgs a) {
  constexpr int R = kFR / C;           // rows whose statistics one CTA owns
  constexpr int TPR = 128 / R;         // owner threads per row
  constexpr int NQ = 16 / TPR;          // 4-column quads per owner thread and 64-column tile
  static_assert(NQ >= 1 && TPR * NQ * 4 == kFV, "owner columns");
  constexpr uint16_t kAll = static_cast<uint16_t>((1u << C) - 1u);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* ring = smem;
  uint8_t* ptiles = smem + kFSmemP;
  uint8_t* parts = smem + kFSmemPart;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kFSmemBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kFSmemMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kFSmemMisc + 4);
  volatile SweepInfo* info = reinterpret_cast<volatile SweepInfo*>(smem + kFSmemMisc + 16);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int cluster = static_cast<int>(blockIdx.x) / C;
  const int num_clusters = static_cast<int>(gridDim.x) / C;
  const int col0 = static_cast<int>(rank) * a.ds;    // first d-column of this CTA's slice

  if (threadIdx.x == 0) {
    for (int i = 0; i < kFStages; ++i) {
      mbar_init(&bars[bWfull + i], 1);
      mbar_init(&bars[bWempty + i], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars[bZfull + b], 1);
      mbar_init(&bars[bZempty + b], 4);
      mbar_init(&bars[bPfull + b], 1);
      mbar_init(&bars[bPfree + b], C);
      mbar_init(&bars[bPartFull + b], 1);
      mbar_init(&bars[bPartFree + b], C);
    }
    mbar_init(&bars[bXready], 4);
    mbar_init(&bars[bOfull], 1);
    mbar_init(&bars[bOempty], 4);
    mbar_init(&bars[bRfull], 1);
    mbar_init(&bars[bDrain], 1);
    *abort_flag = 0;
    fence_mbarrier_init();
    tma_prefetch_desc(&tmW);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();              // every CTA's barriers exist before anyone signals them
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Initial phases: no owner holds partials and no P tile is in use yet, so
  // each CTA completes phase 0 of every CTA's "partials free" and "P free".
  if (threadIdx.x == 192) {
    for (int c = 0; c < C; ++c)
      for (int b = 0; b < 2; ++b) {
        mbar_arrive_remote(map_to_rank(smem_u32(&bars[bPartFree + b]), c));
        mbar_arrive_remote(map_to_rank(smem_u32(&bars[bPfree + b]), c));
      }
    for (int b = 0; b < 2; ++b) mbar_arrive_expect_tx(&bars[bPartFull + b], C * R * kFV * 4);
  }
  if (threadIdx.x == 64) mbar_arrive_expect_tx(&bars[bRfull], kFR * 16);

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t t = 0, issued = 0, last_phase = 0;
      bool ok = true;
      const uint32_t bytes = static_cast<uint32_t>(a.ds) * kFV * 2;
      for (int s = 0; ok; ++s) {
        if (!(ok = mbar_wait(&bars[bXready], s & 1, abort_flag))) break;
        if (!info->valid) break;
        for (int j = 0; j < a.n_tiles; ++j, ++t) {
          const int st = t % kFStages;
          const uint32_t ph = (t / kFStages) & 1;
          if (!(ok = mbar_wait(&bars[bWempty + st], ph ^ 1, abort_flag))) break;
          mbar_arrive_expect_tx(&bars[bWfull + st], bytes);
          for (int at = 0; at < a.ds / 64; ++at)
            tma_load_2d(ring + st * kFStageBytes + at * kFAtom, &tmW, &bars[bWfull + st],
                        col0 + 64 * at, j * kFV);
          issued |= 1u << st;
          last_phase = (last_phase & ~(1u << st)) | (ph << st);
        }
      }
      if (!ok) {
        atomicOr(a.flags, SOLO_FLAG_TIMEOUT);
        for (int st = 0; st < kFStages; ++st)
          if (issued & (1u << st)) drain_wait(&bars[bWfull + st], (last_phase >> st) & 1u);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idz = idesc_bf16_f32(kFR, kFV, false, false);
      const uint32_t ido = idesc_bf16_f32(kFR, a.ds, false, true);
      const uint32_t ring_a = smem_u32(ring), p_a = smem_u32(ptiles);
      uint32_t t = 0;
      bool ok = true;
      // O += P W for tile tt (the j-th of sweep s): P K-major (one atom), the W
      // slice MN-major (atoms of 64 d-columns, kFAtom apart).
      auto issue_o = [&](int j, uint32_t tt, int s) -> bool {
        const int b = tt & 1;
        if (!mbar_wait_cluster(&bars[bPfull + b], (tt >> 1) & 1, abort_flag)) return false;
        if (j == 0 && s > 0 && !mbar_wait(&bars[bOempty], (s - 1) & 1, abort_flag)) return false;
        tc_fence_after();
        const uint32_t sb = ring_a + (tt % kFStages) * kFStageBytes;
        const uint32_t pb = p_a + b * kFPBytes;
#pragma unroll
        for (int k = 0; k < kFV / 16; ++k) {
          const uint64_t ad = smem_desc_sw128(pb + k * 32, 16, 1024);
          const uint64_t bd = smem_desc_sw128(sb + k * 2048, kFAtom, 1024);
          mma_bf16(tmem + kTO, ad, bd, ido, (j > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit_multicast(&bars[bPfree + b], kAll);   // this CTA's P buffer is free again
        mma_commit(&bars[bWempty + tt % kFStages]);
        return true;
      };
      for (int s = 0; ok; ++s) {
        if (!(ok = mbar_wait(&bars[bXready], s & 1, abort_flag))) break;
        if (!info->valid) break;
        tc_fence_after();
        const uint32_t t0 = t;
        for (int j = 0; j < a.n_tiles; ++j, ++t) {
          const int st = t % kFStages, b = t & 1;
          if (!(ok = mbar_wait(&bars[bWfull + st], (t / kFStages) & 1, abort_flag))) break;
          if (t >= 2 && !(ok = mbar_wait(&bars[bZempty + b], ((t >> 1) - 1) & 1, abort_flag))) break;
          tc_fence_after();
          const uint32_t sb = ring_a + st * kFStageBytes;
          // partial Z = xhat slice (tensor memory) x W slice^T (K-major atoms)
          for (int k = 0; k < a.ds / 16; ++k) {
            const uint64_t bd = smem_desc_sw128(sb + (k / 4) * kFAtom + (k % 4) * 32, 16, 1024);
            mma_bf16_ts(tmem + kTZ + b * kFV, tmem + kTX + 8 * k, bd, idz, k > 0 ? 1u : 0u);
          }
          mma_commit(&bars[bZfull + b]);
          // the O product of an earlier tile while this tile's partial Z is exchanged
          if (j >= kFLag && !(ok = issue_o(j - kFLag, t - kFLag, s))) break;
        }
        if (!ok) break;
        const int first = a.n_tiles > kFLag ? a.n_tiles - kFLag : 0;
        for (int j = first; ok && j < a.n_tiles; ++j) ok = issue_o(j, t0 + j, s);
        if (!ok) break;
        mma_commit(&bars[bOfull]);
      }
      if (!ok) {
        atomicOr(a.flags, SOLO_FLAG_TIMEOUT);
        mma_commit(&bars[bDrain]);
        drain_wait(&bars[bDrain], 0);
      }
    }
    __syncwarp();
  } else if (warp < 6) {
    // ------------------------------------------------------------ lane warps
    const int q = warp & 3;                            // tensor-memory lane quadrant
    const uint32_t lanes = static_cast<uint32_t>(32 * q) << 16;
    const int rr = 32 * q + lane;                      // row within the block
    const int owner = rr / R;
    const int ri = rr - owner * R;
    const int prow_src = static_cast<int>(rank) * R + ri;   // row in the owner's buffer
    const uint32_t part_dst = map_to_rank(smem_u32(parts + prow_src * kFV * 4), owner);
    const uint32_t part_bar = map_to_rank(smem_u32(&bars[bPartFull]), owner);
    const int slice_cols = max(0, min(a.ds, a.d - col0));   // valid d-columns of the slice
    uint32_t t = 0;
    bool ok = true;
    int rb = cluster, redo = 0;
    for (int s = 0;; ++s) {
      const int valid = rb < a.row_blocks;
      const int64_t row = static_cast<int64_t>(rb) * kFR + rr;
      if (valid && !redo) {
        // this CTA's slice of xhat for the block, two bf16 per tensor-memory column
        const bool row_ok = row < a.M;
        const uint4* src = reinterpret_cast<const uint4*>(a.xhat + row * a.d + col0);
        for (int c = 0; c < a.ds / 64; ++c) {
          uint32_t w[32];
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int col = 64 * c + 8 * u;
            uint4 x = make_uint4(0, 0, 0, 0);
            if (row_ok && col < slice_cols) x = __ldg(src + (col >> 3));
            w[4 * u] = x.x;
            w[4 * u + 1] = x.y;
            w[4 * u + 2] = x.z;
            w[4 * u + 3] = x.w;
          }
          tmem_st32(tmem + lanes + kTX + 32 * c, w);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (warp == 2 && lane == 0) {
        info->valid = valid;
        info->rb = rb;
        info->redo = redo;
      }
      if (lane == 0) mbar_arrive(&bars[bXready]);
      if (!valid) break;

      for (int j = 0; j < a.n_tiles; ++j, ++t) {
        const int b = t & 1;
        const uint32_t ph = (t >> 1) & 1;
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[bZfull + b], ph, abort_flag) &&
                                         mbar_wait_cluster(&bars[bPartFree + b], ph, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const uint32_t dst = part_dst + b * kFPartBytes;
        const uint32_t bar = part_bar + b * 8;
#pragma unroll 1
        for (int c = 0; c < kFV / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lanes + kTZ + b * kFV + 32 * c, v);
#pragma unroll
          for (int u = 0; u < 8; ++u)
            st_async_v4(dst + (((8 * c + u) ^ (prow_src & 15)) << 4), __float_as_uint(v[4 * u]),
                        __float_as_uint(v[4 * u + 1]), __float_as_uint(v[4 * u + 2]),
                        __float_as_uint(v[4 * u + 3]), bar);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[bZempty + b]);
      }
      if (!ok) break;

      // end of the sweep: O is complete and the owners' per-row factors are in
      // the first 2 KB of P buffer t & 1 (16 B per row: a, b, coef, overflow bits)
      ok = __all_sync(0xffffffffu, mbar_wait(&bars[bOfull], s & 1, abort_flag) &&
                                       mbar_wait_cluster(&bars[bRfull], s & 1, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const float4* rowfac = reinterpret_cast<const float4*>(ptiles + (t & 1) * kFPBytes);
      uint32_t over = 0;
#pragma unroll
      for (int u = 0; u < 4; ++u) over |= __float_as_uint(rowfac[lane + 32 * u].w);
      const bool redo_next = !redo && __any_sync(0xffffffffu, over != 0u);
      const float4 f = rowfac[rr];
      __syncwarp();
      if (warp == 2 && lane == 0) mbar_arrive_expect_tx(&bars[bRfull], kFR * 16);
      if (!redo_next && slice_cols > 0) {
        // dH = r gamma dxhat - coef h with dxhat = a O - b W_y (the final RMSNorm's
        // backward, as in the dX̂ GEMM's epilogue of the stored path)
        const bool row_ok = row < a.M;
        int k = 0;
        int64_t n = 0;
        int y = -1;
        float rn = 0.f;
        if (row_ok) {
          k = static_cast<int>(row / a.N);
          n = row - static_cast<int64_t>(k) * a.N;
          y = a.targets[row];
          rn = a.r[row];
        }
        const bool use_wy = row_ok && f.y != 0.f && y >= 0 && y < a.V;
        const bool mod_ok = row_ok && in_bounds(k < a.modules, a.flags);
        for (int c = 0; c * 32 < slice_cols; ++c) {
          float o[32];
          tmem_ld32(tmem + lanes + kTO + 32 * c, o);
          if (!mod_ok) continue;
          const int cbase = col0 + 32 * c;
          const uint16_t* hrow = a.hidden[k] + n * a.d;
          uint16_t* dhrow = a.dhidden[k] + n * a.d;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int col = cbase + 8 * u;
            if (col >= a.d || 32 * c + 8 * u >= a.ds) break;
            const uint4 hv = __ldg(reinterpret_cast<const uint4*>(hrow + col));
            const uint4 gv = __ldg(reinterpret_cast<const uint4*>(a.gamma + col));
            uint4 wv = make_uint4(0, 0, 0, 0);
            if (use_wy)
              wv = __ldg(reinterpret_cast<const uint4*>(a.W + static_cast<int64_t>(y) * a.d + col));
            const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
            const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w};
            const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
            uint32_t outw[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float x0 = fmaf(f.x, o[8 * u + 2 * e], -f.y * bf_lo(ww[e]));
              const float x1 = fmaf(f.x, o[8 * u + 2 * e + 1], -f.y * bf_hi(ww[e]));
              outw[e] = pack_bf16x2(fmaf(rn * bf_lo(gw[e]), x0, -f.z * bf_lo(hw[e])),
                                    fmaf(rn * bf_hi(gw[e]), x1, -f.z * bf_hi(hw[e])));
            }
            *reinterpret_cast<uint4*>(dhrow + col) = make_uint4(outw[0], outw[1], outw[2], outw[3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[bOempty]);
      if (redo_next) {
        redo = 1;
      } else {
        redo = 0;
        rb += num_clusters;
      }
    }
    if (!ok && lane == 0) atomicOr(a.flags, SOLO_FLAG_TIMEOUT);
  } else {
    // ------------------------------------------------------------ owners
    const int ot = static_cast<int>(threadIdx.x) - 192;
    const int i = ot / TPR;                    // row among this CTA's R rows
    const int g = ot - i * TPR;                // column group of the row
    const int prow = static_cast<int>(rank) * R + i;   // row of the P tile
    uint32_t t = 0;
    bool ok = true;
    float m_exact = -INFINITY;
    for (int s = 0;; ++s) {
      ok = named_bar_and(1, 128, mbar_wait(&bars[bXready], s & 1, abort_flag));
      if (!ok) break;
      const int valid = info->valid, rb = info->rb, redo = info->redo;
      if (!valid) break;
      const int64_t row = static_cast<int64_t>(rb) * kFR + prow;
      const bool row_ok = row < a.M;
      int y = -1, kmod = 0;
      bool kept = false;
      float rn = 0.f;
      if (row_ok) {
        y = a.targets[row];
        kept = row_kept(a, row, y);
        kmod = static_cast<int>(row / a.N);
        rn = a.r[row];
      }
      if (!redo) m_exact = -INFINITY;
      float mref = redo ? m_exact : 0.f;
      float S = 0.f, U = 0.f, zy = 0.f;
      bool over = false;
      for (int j = 0; j < a.n_tiles; ++j, ++t) {
        const int b = t & 1;
        const uint32_t ph = (t >> 1) & 1;
        ok = named_bar_and(1, 128, mbar_wait_cluster(&bars[bPartFull + b], ph, abort_flag));
        if (!ok) break;
        // z = sum of the C partials, in rank order.  The row's 64 columns are 16
        // quads of 4; thread g of the row takes quads g, g + TPR, ...
        const float* prt = reinterpret_cast<const float*>(parts + b * kFPartBytes);
        float z[NQ][4];
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
          const int qd = g + TPR * m;
          // row src * R + i of the buffer; (src * R + i) & 15 == i & 15 since R >= 16
          const int pos = 4 * (qd ^ (i & 15));
          float4 acc = *reinterpret_cast<const float4*>(prt + i * kFV + pos);
#pragma unroll
          for (int src = 1; src < C; ++src) {
            const float4 x = *reinterpret_cast<const float4*>(prt + (src * R + i) * kFV + pos);
            acc.x += x.x;
            acc.y += x.y;
            acc.z += x.z;
            acc.w += x.w;
          }
          z[m][0] = acc.x;
          z[m][1] = acc.y;
          z[m][2] = acc.z;
          z[m][3] = acc.w;
        }
        // the partials are consumed (the loads completed at the barrier): arm the
        // buffer's next phase and tell every source, one owner thread per source
        named_bar_and(2, 128, true);
        if (ot == 0) mbar_arrive_expect_tx(&bars[bPartFull + b], C * R * kFV * 4);
        if (ot < C) mbar_arrive_remote_relaxed(map_to_rank(smem_u32(&bars[bPartFree + b]), ot));
        const int cbase = j * kFV;
        float tmax = -INFINITY;
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
          const int qd = g + TPR * m;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            if (cbase + 4 * qd + e >= a.V) z[m][e] = -INFINITY;   // past the vocabulary
            tmax = fmaxf(tmax, z[m][e]);
          }
        }
#pragma unroll
        for (int o = 1; o < TPR; o <<= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
        m_exact = fmaxf(m_exact, tmax);
        if (!redo) {
          if (j == 0) mref = tmax;
          else if (kept && tmax > mref + kMoveRef) over = true;
        }
        // the target's own term is left out of S, U and P; its logit is kept
        const int yrel = kept ? y - cbase : -1;
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
          const int qd = g + TPR * m;
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if (4 * qd + e == yrel) {
              zy = z[m][e];
              z[m][e] = -INFINITY;
            }
        }
        // every CTA's product of the buffer's previous tile is done: it is free
        ok = named_bar_and(1, 128, mbar_wait_cluster(&bars[bPfree + b], ph, abort_flag));
        if (!ok) break;
        uint8_t* ptile = ptiles + b * kFPBytes;
        const bool live = kept && !over;
        const float ml = mref * kLog2e;
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
          float e4[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            e4[e] = live ? ex2_approx(fmaf(z[m][e], kLog2e, -ml)) : 0.f;
            S += e4[e];
            U += e4[e] > 0.f ? e4[e] * z[m][e] : 0.f;
          }
          // quad qd = half of the 16-byte chunk qd / 2 of the (swizzled) P row
          const int qd = g + TPR * m;
          const uint32_t addr =
              smem_u32(ptile + prow * 128 + ((((qd >> 1) ^ (prow & 7)) << 4) | ((qd & 1) << 3)));
          asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr),
                       "r"(pack_bf16x2(e4[0], e4[1])), "r"(pack_bf16x2(e4[2], e4[3]))
                       : "memory");
        }
        fence_proxy_async_smem();
        named_bar_and(2, 128, true);
        // this CTA's R rows of P to every other CTA of the cluster, one owner
        // thread per peer
        if (ot < C - 1) {
          const uint32_t off = b * kFPBytes + static_cast<int>(rank) * R * 128;
          const uint32_t peer = (rank + 1 + ot) % C;
          bulk_copy_s2s(map_to_rank(smem_u32(ptiles + off), peer), smem_u32(ptiles + off),
                        R * 128, map_to_rank(smem_u32(&bars[bPfull + b]), peer));
        }
        if (ot == C - 1) mbar_arrive_expect_tx(&bars[bPfull + b], (C - 1) * R * 128);
      }
      if (!ok) break;
      // ---- end of the sweep: the row's totals over its TPR threads
      float zyt = zy;
#pragma unroll
      for (int o = 1; o < TPR; o <<= 1) {
        S += __shfl_xor_sync(0xffffffffu, S, o);
        U += __shfl_xor_sync(0xffffffffu, U, o);
        zyt += __shfl_xor_sync(0xffffffffu, zyt, o);   // one thread of the row holds z_y
      }
      float fa = 0.f, fb = 0.f, fcoef = 0.f, loss = 0.f;
      if (kept && !over) {
        // lse - z_y without cancellation (the target's term is not in S)
        const float dy = zyt - mref;
        const float nll = dy >= 0.f ? log1pf(S * expf(-dy)) : -dy + logf(S + expf(dy));
        const float inv_s = expf(-(nll + dy));            // 1 / (S' + e^{z_y - m}) = e^{m - lse}
        const float w = a.inv_nvalid[kmod];
        const float edz = (U - zyt * S) * inv_s;          // E_p[z] - z_y
        fa = w * inv_s;
        fb = w * -expm1f(-nll);                           // (1 - p_y) / Nvalid
        fcoef = rn * rn * (w * edz) / static_cast<float>(a.d);
        loss = nll;
      }
      if (row_ok && g == 0) {
        if (a.loss_tok) a.loss_tok[row] = loss;
        a.row_loss[row] = loss;
      }
      // P buffer t & 1 (its last user, tile t - 2, is done everywhere) carries the
      // factors; the next sweep's owners write it only after every CTA's lanes
      // have read them (their partials of that sweep come after)
      ok = named_bar_and(1, 128, mbar_wait_cluster(&bars[bPfree + (t & 1)], (t >> 1) & 1, abort_flag));
      if (!ok) break;
      if (g == 0) {
        const uint32_t ob = over ? 1u : 0u;
        const uint32_t dst = smem_u32(ptiles + (t & 1) * kFPBytes + prow * 16);
#pragma unroll 1
        for (int c = 0; c < C; ++c)
          st_async_v4(map_to_rank(dst, c), __float_as_uint(fa), __float_as_uint(fb),
                      __float_as_uint(fcoef), ob, map_to_rank(smem_u32(&bars[bRfull]), c));
      }
    }
    if (!ok && ot == 0) atomicOr(a.flags, SOLO_FLAG_TIMEOUT);
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();              // no CTA leaves while a peer may still write to it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Kept-token counts of the auxiliary modules, 1/Nvalid, bad-target flags.
__global__ void __launch_bounds__(256) flash_count_kernel(const FlashArgs a, float* inv_nvalid) {
  const int k = blockIdx.x;
  int c = 0, bad = 0;
  for (int64_t n = threadIdx.x; n < a.N; n += 256) {
    const int64_t row = static_cast<int64_t>(k) * a.N + n;
    const int y = a.targets[row];
    const bool in = y >= 0 && y < a.V;
    bad |= (!in && y != a.ignore_index) ? 1 : 0;
    c += row_kept(a, row, y) ? 1 : 0;
  }
  __shared__ int sc[256];
  sc[threadIdx.x] = c;
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(a.flags, SOLO_FLAG_BAD_TARGET);
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) sc[threadIdx.x] += sc[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    a.n_valid[k] = sc[0];
    inv_nvalid[k] = sc[0] > 0 ? static_cast<float>(1.0 / static_cast<double>(sc[0])) : 0.f;
  }
}

// loss_mean[k] = (sum of the module's token losses) / Nvalid, fixed order.
__global__ void __launch_bounds__(256) flash_means_kernel(const FlashArgs a) {
  const int k = blockIdx.x;
  double s = 0.0;
  for (int64_t n = threadIdx.x; n < a.N; n += 256) s += a.row_loss[static_cast<int64_t>(k) * a.N + n];
  __shared__ double sd[256];
  sd[threadIdx.x] = s;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) sd[threadIdx.x] += sd[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int nv = a.n_valid[k];
    a.loss_mean[k] = nv > 0 ? static_cast<float>(sd[0] / static_cast<double>(nv)) : 0.f;
  }
}

template <int C>
cudaError_t set_attr() {
  return cudaFuncSetAttribute(flash_bwd_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kFSmemTotal);
}

template <int C>
int active_clusters() {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(C, 1, 1);
  cfg.blockDim = dim3(kFThreads, 1, 1);
  cfg.dynamicSmemBytes = kFSmemTotal;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, flash_bwd_kernel<C>, &cfg) != cudaSuccess) return 0;
  return n;
}

std::mutex g_flash_mu;
int g_flash_clusters[64][4];   // per device: co-resident clusters for C = 1, 2, 4, 8

}  // namespace

cudaError_t flash_prepare(int device) {
  if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
  cudaError_t e = set_attr<1>();
  if (e == cudaSuccess) e = set_attr<2>();
  if (e == cudaSuccess) e = set_attr<4>();
  if (e == cudaSuccess) e = set_attr<8>();
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_flash_mu);
  g_flash_clusters[device][0] = active_clusters<1>();
  g_flash_clusters[device][1] = active_clusters<2>();
  g_flash_clusters[device][2] = active_clusters<4>();
  g_flash_clusters[device][3] = active_clusters<8>();
  cudaGetLastError();
  return cudaSuccess;
}

cudaError_t launch_flash_count(const FlashArgs& a, float* inv_nvalid, cudaStream_t s) {
  if (a.modules <= 0) return cudaSuccess;
  flash_count_kernel<<<a.modules, 256, 0, s>>>(a, inv_nvalid);
  return launched();
}

cudaError_t launch_flash_means(const FlashArgs& a, cudaStream_t s) {
  if (a.modules <= 0) return cudaSuccess;
  flash_means_kernel<<<a.modules, 256, 0, s>>>(a);
  return launched();
}

cudaError_t launch_flash(const CUtensorMap& w, const FlashArgs& a, int device, int sms,
                         cudaStream_t s) {
  if (a.M <= 0) return cudaSuccess;
  const int C = flash_cluster_size(a.d);
  const int ci = C == 1 ? 0 : C == 2 ? 1 : C == 4 ? 2 : 3;
  int fit = 0;
  {
    std::lock_guard<std::mutex> lock(g_flash_mu);
    fit = (device >= 0 && device < 64) ? g_flash_clusters[device][ci] : 0;
  }
  if (fit <= 0) fit = std::max(1, sms / C);
  const int clusters = std::min(a.row_blocks, fit);
  const dim3 grid(static_cast<unsigned>(C * clusters));
  switch (C) {
    case 1: flash_bwd_kernel<1><<<grid, kFThreads, kFSmemTotal, s>>>(w, a); break;
    case 2: flash_bwd_kernel<2><<<grid, kFThreads, kFSmemTotal, s>>>(w, a); break;
    case 4: flash_bwd_kernel<4><<<grid, kFThreads, kFSmemTotal, s>>>(w, a); break;
    default: flash_bwd_kernel<8><<<grid, kFThreads, kFSmemTotal, s>>>(w, a); break;
  }
  return launched();
}

int flash_cluster_size(int d) { return d <= 256 ? 1 : d <= 512 ? 2 : d <= 1024 ? 4 : 8; }

int flash_slice_width(int d) {
  const int c = flash_cluster_size(d);
  return ((d + c - 1) / c + 63) / 64 * 64;
}

}  // namespace solo
