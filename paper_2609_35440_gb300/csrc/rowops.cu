// Row-wise kernels of the readout path: the final RMSNorm, the log-sum-exp
// combination of per-tile statistics with the token loss and module means, the
// gradient of the logits, and the dgamma reduction.  (The RMSNorm backward runs
// in the epilogue of the dX̂ GEMM.)
//
// All reductions run in a fixed order (no floating-point atomics), so every
// output is bitwise reproducible from run to run.
#include <cuda_bf16.h>

#include "internal.h"
#include "../../include/solo_readout.h"

namespace solo {
namespace {

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&b);
}

__device__ __forceinline__ void unpack8(const uint4& x, float (&f)[8]) {
  f[0] = bf16_lo(x.x); f[1] = bf16_hi(x.x);
  f[2] = bf16_lo(x.y); f[3] = bf16_hi(x.y);
  f[4] = bf16_lo(x.z); f[5] = bf16_hi(x.z);
  f[6] = bf16_lo(x.w); f[7] = bf16_hi(x.w);
}

__device__ __forceinline__ bool token_kept(const RowArgs& a, int64_t row, int y) {
  const bool in_range = y >= 0 && y < a.V;
  return in_range && y != a.ignore_index && (a.mask == nullptr || a.mask[row] != 0);
}

// ---- kept-token compaction ------------------------------------------------------
// Masked tokens need no logits and no gradient: the kept ones take rows
// [0, Mk) of every per-row buffer (token order, module by module), so the
// products run over Mk rows only.  Ranks are exact integer prefix sums: the
// compact order is the token order, whatever the schedule.

// Per chunk of kScanRows tokens of module blockIdx.y: each token's count of kept
// tokens before it within the chunk, and the chunk's total; bad targets flagged.
__global__ void __launch_bounds__(kScanRows) keep_scan_kernel(const RowArgs a) {
  __shared__ int warp_tot[kScanRows / 32];
  const int k = blockIdx.y;
  const int64_t n = static_cast<int64_t>(blockIdx.x) * kScanRows + threadIdx.x;
  const int64_t row = static_cast<int64_t>(k) * a.N + n;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int kept = 0, bad = 0;
  if (n < a.N) {
    const int y = a.targets[row];
    kept = token_kept(a, row, y) ? 1 : 0;
    bad = (!(y >= 0 && y < a.V) && y != a.ignore_index) ? 1 : 0;
  }
  const uint32_t ballot = __ballot_sync(0xffffffffu, kept);
  const int in_warp = __popc(ballot & ((1u << lane) - 1u));
  if (lane == 0) warp_tot[warp] = __popc(ballot);
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(a.flags, SOLO_FLAG_BAD_TARGET);
  if (warp == 0) {
    const int v = warp_tot[lane];          // kScanRows / 32 == 32 warps
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int x = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += x;
    }
    warp_tot[lane] = incl - v;             // exclusive prefix of the warp totals
    if (lane == 31) a.chunk_base[static_cast<int64_t>(k) * a.nchunks + blockIdx.x] = incl;
  }
  __syncthreads();
  if (n < a.N) a.kept_local[row] = warp_tot[warp] + in_warp;
}

// One block: chunk counts -> exclusive prefix over (module, chunk) in order;
// offsets[k] = first compact row of module k, offsets[K] = Mk.
__global__ void __launch_bounds__(1024) keep_offsets_kernel(const RowArgs a) {
  __shared__ int warp_sum[32];
  __shared__ int carry_s;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t total = static_cast<int64_t>(a.K) * a.nchunks;
  if (threadIdx.x == 0) carry_s = 0;
  __syncthreads();
  for (int64_t base = 0; base < total; base += 1024) {
    const int64_t i = base + threadIdx.x;
    const int v = i < total ? a.chunk_base[i] : 0;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int x = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += x;
    }
    if (lane == 31) warp_sum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int w = warp_sum[lane];
      int wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += x;
      }
      warp_sum[lane] = wi - w;
    }
    __syncthreads();
    const int carry = carry_s;
    if (i < total) {
      const int ex = carry + warp_sum[warp] + incl - v;
      a.chunk_base[i] = ex;
      if (i % a.nchunks == 0) a.offsets[i / a.nchunks] = ex;
    }
    __syncthreads();
    if (threadIdx.x == 1023) carry_s = carry + warp_sum[warp] + incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    a.offsets[a.K] = carry_s;
    if (a.grad_count) *a.grad_count = 0;   // the gradient pass's row list starts empty
  }
}

// ---- final RMSNorm: r_i = (mean_j h_ij^2 + eps)^-1/2, xhat = bf16(gamma h r) ------
// The bf16 rounding of xhat is a quantisation decision, so it is taken on the
// exact value, in fp32 arithmetic only (fp64 is slow on this part):
//  - the sum of squares is accumulated error-free: each h^2 of a bf16 h is
//    exact in fp32 and TwoSum keeps the rounding error of every addition
//    (eight independent chains per lane, then pairwise across the warp), so
//    the row's sum is an unevaluated pair (hi, lo) accurate to ~2^-46;
//  - r = (ss/d + eps)^-1/2 comes from rsqrtf refined by one Newton step whose
//    residual 1 - x r0^2 is formed with exact products (FMA), giving r as a
//    pair (r32, r_lo) accurate to ~2^-44;
//  - y = gamma h r is rounded from fp32 when it lies more than 4 ulp from a
//    bf16 midpoint (|fl(gamma h r32) - y| <= 2 ulp); otherwise the sign of
//    (y - midpoint) is decided from the exact product gamma h (r32 + r_lo).

struct F2 {
  float hi, lo;
};

__device__ __forceinline__ F2 two_sum(float a, float b) {
  const float s = a + b;
  const float bb = s - a;
  return {s, (a - (s - bb)) + (b - bb)};
}

// (a.hi + a.lo) + (b.hi + b.lo), renormalised
__device__ __forceinline__ F2 add_f2(F2 a, F2 b) {
  const F2 s = two_sum(a.hi, b.hi);
  const float lo = s.lo + a.lo + b.lo;
  const float hi = s.hi + lo;
  return {hi, lo - (hi - s.hi)};
}

// (r32 + r_lo) ~= (x.hi + x.lo)^-1/2
__device__ __forceinline__ F2 rsqrt_f2(F2 x) {
  const float r0 = rsqrtf(x.hi);
  const float q_hi = r0 * r0;
  const float q_lo = fmaf(r0, r0, -q_hi);                // r0^2 = q_hi + q_lo exactly
  const float p_hi = x.hi * q_hi;
  const float p_lo = fmaf(x.hi, q_hi, -p_hi) + fmaf(x.hi, q_lo, x.lo * q_hi);
  const float e = (1.0f - p_hi) - p_lo;                  // 1 - x r0^2 (tiny)
  const float corr = 0.5f * r0 * e;                      // Newton: r = r0 (1 + e/2)
  const float r32 = r0 + corr;
  return {r32, corr - (r32 - r0)};
}

__device__ __forceinline__ uint16_t xhat_bf16(float gh, F2 r) {
  const float y = gh * r.hi;          // gh = gamma * h is exact in fp32
  const uint32_t b = __float_as_uint(y);
  const uint32_t mag = b & 0x7FFFFFFFu;
  const int low = static_cast<int>(mag & 0xFFFFu) - 0x8000;
  if (low >= -4 && low <= 4 && mag < 0x7F000000u && mag >= 0x00800000u) {
    // The exact value lies strictly between the two neighbouring bf16
    // values; compare it with their midpoint.
    const uint32_t down = mag & 0xFFFF0000u;
    const float mid = __uint_as_float(down | 0x8000u);
    const float ga = fabsf(gh);
    const float p_hi = ga * r.hi;
    const float p_lo = fmaf(ga, r.hi, -p_hi) + ga * r.lo; // ga * (r.hi + r.lo) = p_hi + p_lo
    const float dmid = (p_hi - mid) + p_lo;                // p_hi - mid is exact (close values)
    uint32_t q = down >> 16;
    if (dmid > 0.f || (dmid == 0.f && (q & 1u))) q += 1;
    return static_cast<uint16_t>(q | ((b >> 16) & 0x8000u));
  }
  return static_cast<uint16_t>((b + 0x7FFFu + ((b >> 16) & 1u)) >> 16);
}

// True when fp32 y lies within 4 ulp of a bf16 midpoint (|low 16 bits - 0x8000| <= 4).
__device__ __forceinline__ bool near_midpoint(float y) {
  return ((__float_as_uint(y) - 0x7FFCu) & 0xFFFFu) <= 8u;
}

// Two x-hat values: away from midpoints the fp32 product rounds like the exact
// value, and the hardware's round-to-nearest-even packs both; otherwise each
// takes the exact test of xhat_bf16.
__device__ __forceinline__ uint32_t xhat_bf16x2(float gh0, float gh1, F2 r) {
  const float y0 = gh0 * r.hi;
  const float y1 = gh1 * r.hi;
  if (near_midpoint(y0) || near_midpoint(y1))
    return static_cast<uint32_t>(xhat_bf16(gh0, r)) |
           (static_cast<uint32_t>(xhat_bf16(gh1, r)) << 16);
  uint32_t w;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w) : "f"(y1), "f"(y0));
  return w;
}

// VPL > 0: the row is held in registers (VPL 16-byte vectors per lane, d <=
// 256 * VPL), so h is read from memory once.  VPL == 0: any d, h re-read.
template <int VPL>
__global__ void __launch_bounds__(256, 4) rmsnorm_fwd_kernel(const RowArgs a) {
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const int lane = threadIdx.x & 31;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  if (row >= M) return;
  const int k = static_cast<int>(row / a.N);
  const int64_t n = row - static_cast<int64_t>(k) * a.N;
  const uint4* h = reinterpret_cast<const uint4*>(a.hidden[k] + n * a.d);
  const uint4* g = reinterpret_cast<const uint4*>(a.gamma);
  const int nv = a.d / 8;
  int64_t out_row = row;
  if (a.kept_local != nullptr) {
    // compact row: kept tokens before this one
    const int64_t before = a.chunk_base[static_cast<int64_t>(k) * a.nchunks + n / kScanRows] +
                           a.kept_local[row];
    const int y = a.targets[row];
    if (!token_kept(a, row, y)) {
      // masked: its loss and dH row are zero, and it zeroes one row of [Mk, M)
      // (the rows past the kept ones that the products read in their last tiles)
      const int64_t slot = a.offsets[a.K] + (row - before);
      uint4* xz = reinterpret_cast<uint4*>(a.xhat + slot * a.d);
      uint4* dz = a.dhidden[k] ? reinterpret_cast<uint4*>(a.dhidden[k] + n * a.d) : nullptr;
      for (int v = lane; v < nv; v += 32) {
        if (in_bounds(slot < M, a.flags)) xz[v] = make_uint4(0, 0, 0, 0);
        if (dz) dz[v] = make_uint4(0, 0, 0, 0);
      }
      if (lane == 0 && a.loss_tok) a.loss_tok[row] = 0.f;
      return;
    }
    out_row = before;
    if (lane == 0 && in_bounds(before < M, a.flags)) {
      a.orig_row[before] = static_cast<int32_t>(row);
      a.tgt_c[before] = y;
    }
  }
  constexpr int kCache = VPL > 0 ? VPL : 1;
  uint4 hc[kCache];
  // eight independent error-free sums (one per element position of a vector)
  float s[8], c[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) s[j] = c[j] = 0.f;
  auto accumulate = [&](const uint4& x) {
    float f[8];
    unpack8(x, f);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float sq = f[j] * f[j];
      const float t = s[j] + sq;
      const float bb = t - s[j];
      c[j] += (s[j] - (t - bb)) + (sq - bb);
      s[j] = t;
    }
  };
  if constexpr (VPL > 0) {
#pragma unroll
    for (int u = 0; u < VPL; ++u) {
      const int v = lane + 32 * u;
      hc[u] = v < nv ? __ldg(h + v) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < VPL; ++u) accumulate(hc[u]);
  } else {
    for (int v = lane; v < nv; v += 32) accumulate(__ldg(h + v));
  }
  F2 ss = {s[0], c[0]};
#pragma unroll
  for (int j = 1; j < 8; ++j) ss = add_f2(ss, F2{s[j], c[j]});
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const F2 other = {__shfl_xor_sync(0xffffffffu, ss.hi, o),
                      __shfl_xor_sync(0xffffffffu, ss.lo, o)};
    ss = add_f2(ss, other);
  }
  // x = ss / d + eps as a pair
  const float fd = static_cast<float>(a.d);
  const float m_hi = ss.hi / fd;
  const float m_lo = (fmaf(-m_hi, fd, ss.hi) + ss.lo) / fd;
  const F2 x = add_f2(F2{m_hi, m_lo}, F2{a.eps, 0.f});
  const F2 rr = rsqrt_f2(x);
  const float r = rr.hi;
  uint4* out = reinterpret_cast<uint4*>(a.xhat + out_row * a.d);
  auto emit = [&](int v, const uint4& x) {
    float f[8], gg[8];
    unpack8(x, f);
    unpack8(__ldg(g + v), gg);
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      w[j] = xhat_bf16x2(gg[2 * j] * f[2 * j], gg[2 * j + 1] * f[2 * j + 1], rr);
    out[v] = make_uint4(w[0], w[1], w[2], w[3]);
  };
  if constexpr (VPL > 0) {
#pragma unroll
    for (int u = 0; u < VPL; ++u) {
      const int v = lane + 32 * u;
      if (v < nv) emit(v, hc[u]);
    }
  } else {
    for (int v = lane; v < nv; v += 32) emit(v, __ldg(h + v));
  }
  if (lane == 0 && a.r) a.r[out_row] = r;
}

// ---- log-sum-exp over column tiles, token loss, per-block module sums ----------

enum LseKind { kLseTrain = 0, kLseExit = 1, kLseHeads = 2 };

// tiles whose statistics one thread loads together (independent loads in flight)
constexpr int kLseBatch = 16;

// kLseExit: also the first argmax over the vocabulary and its log-probability;
// targets may be absent (decoding only).  kLseHeads: also the temperature's
// gradient term E_p[s] - s_y of every kept token (s: logits before the
// temperature and bias), summed per module like the loss.
template <int kKind>
__global__ void __launch_bounds__(256) lse_kernel(const RowArgs a) {
  constexpr bool kExit = kKind == kLseExit;
  constexpr bool kHeads = kKind == kLseHeads;
  const int k = blockIdx.y;
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const int64_t n = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
  // compacted: the module's kept tokens are rows [offsets[k], offsets[k + 1])
  const bool compact = a.kept_local != nullptr;
  const int64_t row = compact ? a.offsets[k] + n : static_cast<int64_t>(k) * a.N + n;
  const bool in_module = compact ? row < a.offsets[k + 1] : n < a.N;
  double lsum = 0.0, tsum = 0.0;
  int cnt = 0;
  int bad = 0;
  if (in_module) {
    const int64_t tok = compact ? a.orig_row[row] : row;     // the token's row of loss_tok
    const int* tgt = compact ? a.tgt_c : a.targets;
    float mx = -INFINITY, s = 0.f, us = 0.f;
    int best_tile = 0;
    bool own_ref = false;       // a tile stored against its own maximum, not 0
    // E_p[s] - s_y = e^{M - lse} sum_t e^{m_t - M} (u_t - s_y s_t), with the
    // target's term left out of the tile sums s_t and u_t = sum of exp(z - m_t) s
    float ys = 0.f;
    if constexpr (!kExit) {
      const int y0 = tgt ? tgt[row] : a.ignore_index;
      if (compact || token_kept(a, row, y0)) ys = kHeads ? a.sy[row] : a.zy[row];
    }
    for (int t0 = 0; t0 < a.n_tiles_v; t0 += kLseBatch) {
      float2 st[kLseBatch];
      float uu[kLseBatch];
#pragma unroll
      for (int u = 0; u < kLseBatch; ++u) {       // independent loads, issued together
        const bool in = t0 + u < a.n_tiles_v;
        st[u] = in ? a.stats[static_cast<int64_t>(t0 + u) * M + row] : make_float2(-INFINITY, 0.f);
        if constexpr (!kExit) uu[u] = in ? a.usum[static_cast<int64_t>(t0 + u) * M + row] : 0.f;
      }
      float cm = mx;
#pragma unroll
      for (int u = 0; u < kLseBatch; ++u) {
        if (kExit && st[u].x > cm) best_tile = t0 + u;   // strict: the first tile with the max
        cm = fmaxf(cm, st[u].x);
        if (!kExit && t0 + u < a.n_tiles_v && st[u].x != 0.f) own_ref = true;
      }
      const float rescale = expf(mx - cm);  // mx = -inf only before the first tile (s = 0)
      s *= rescale;
      if constexpr (!kExit) us *= rescale;
#pragma unroll
      for (int u = 0; u < kLseBatch; ++u) {
        const float f = expf(st[u].x - cm);
        s += st[u].y * f;
        if constexpr (!kExit) {
          us += fmaf(-ys, st[u].y, uu[u]) * f;   // padding tiles add 0: f = 0, s_t = u_t = 0
        }
      }
      mx = cm;
    }
    const int y = tgt ? tgt[row] : a.ignore_index;
    bad = !compact && !(y >= 0 && y < a.V) && y != a.ignore_index;
    const bool kept = compact || token_kept(a, row, y);
    float l = mx + logf(s), nll = 0.f;
    if constexpr (kExit) {
      if (a.top1 && in_bounds(best_tile < a.n_tiles_v, a.flags))
        a.top1[row] = a.argmax[static_cast<int64_t>(best_tile) * M + row];
      if (a.top1_logprob) a.top1_logprob[row] = mx - l;
      nll = l - a.zy[row];
    } else {
      if (y >= 0 && y < a.V) {
        // the tile sums leave the target's term out: lse - z_y without
        // cancellation.  u = sum over v != y of e^{z_v - z_y} (inf when it
        // overflows).  While u <= 1 (p_y >= 1/2) log1p(u) keeps 1 - p_y's
        // relative precision, whatever the reference mx is: it is 0 for the
        // tiles whose logits stay within +-64, so a confident target may lie
        // below it.  Otherwise lse - z_y >= ln 2 and the second form does not
        // cancel.
        const float zt = a.zy[row];
        const float u = s > 0.f ? s * expf(mx - zt) : 0.f;
        nll = (zt >= mx || u <= 1.f) ? log1pf(u) : (mx - zt) + logf(s + expf(zt - mx));
        l = zt + nll;
        a.nll[row] = nll;
      }
      a.lse[row] = l;
    }
    const float loss = kept ? nll : 0.f;
    if (a.loss_tok) a.loss_tok[tok] = loss;
    lsum = loss;
    cnt = kept ? 1 : 0;
    if constexpr (!kExit) {
      // E_p[s] - s_y (s: the logits before temperature and bias; s = z
      // without them): the temperature's gradient term and, scaled, the
      // RMSNorm backward's row sum
      const float e = kept ? us * expf(mx - l) : 0.f;   // the sums are relative to mx
      a.edz[row] = e;
      if constexpr (kHeads) tsum = e;
      if (a.row_fa != nullptr) {
        // A row whose tiles all used the reference 0: its gradient is
        // tau/Nvalid (e^{-lse} P - (1 - p_y) e_y) with P the stored exponentials
        // (e^{-lse} kept well inside fp32 by lse <= 60).  An auxiliary row's is
        // formed by the dX̂ epilogue (fb = 1 - p_y: the W_y term).  A final-module
        // row's target entry of P becomes -(1 - p_y) e^{lse} in the gradient
        // pass, so that tau/Nvalid e^{-lse} P is its whole G row (fb = 0).  The
        // gradient pass turns P into G for the other rows (and sums every row
        // when bias gradients are wanted).
        const int kk = static_cast<int>(tok / a.N);
        const bool factor = kept && !own_ref && l <= 60.f;
        a.row_fa[row] = factor ? expf(-l) : -1.f;
        a.row_fb[row] = (factor && kk < a.K - 1) ? -expm1f(-nll) : 0.f;
      }
    }
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(a.flags, SOLO_FLAG_BAD_TARGET);
  __shared__ double ssum[8], stau[8];
  __shared__ int scnt[8];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
    cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    if constexpr (kHeads) tsum += __shfl_xor_sync(0xffffffffu, tsum, o);
  }
  if ((threadIdx.x & 31) == 0) {
    ssum[threadIdx.x >> 5] = lsum;
    scnt[threadIdx.x >> 5] = cnt;
    stau[threadIdx.x >> 5] = tsum;
  }
  __syncthreads();
  if (threadIdx.x == 0 &&
      in_bounds(k < a.K && static_cast<int>(blockIdx.x) < a.part_blocks, a.flags)) {
    double t = 0.0, tt = 0.0;
    int c = 0;
    for (int w = 0; w < 8; ++w) {
      t += ssum[w];
      c += scnt[w];
      tt += stau[w];
    }
    a.part_sum[static_cast<int64_t>(k) * a.part_blocks + blockIdx.x] = t;
    a.part_cnt[static_cast<int64_t>(k) * a.part_blocks + blockIdx.x] = c;
    if constexpr (kHeads) a.part_tau[static_cast<int64_t>(k) * a.part_blocks + blockIdx.x] = tt;
  }
}

__global__ void __launch_bounds__(256) module_mean_kernel(const RowArgs a) {
  const int k = blockIdx.x;
  double t = 0.0, tt = 0.0;
  long long c = 0;
  for (int b = threadIdx.x; b < a.part_blocks; b += 256) {
    t += a.part_sum[static_cast<int64_t>(k) * a.part_blocks + b];
    c += a.part_cnt[static_cast<int64_t>(k) * a.part_blocks + b];
    if (a.dtau) tt += a.part_tau[static_cast<int64_t>(k) * a.part_blocks + b];
  }
  __shared__ double st[256], stt[256];
  __shared__ long long sc[256];
  st[threadIdx.x] = t;
  sc[threadIdx.x] = c;
  stt[threadIdx.x] = tt;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) {
      st[threadIdx.x] += st[threadIdx.x + o];
      sc[threadIdx.x] += sc[threadIdx.x + o];
      stt[threadIdx.x] += stt[threadIdx.x + o];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const long long nv = sc[0];
    if (a.loss_mean)
      a.loss_mean[k] = nv > 0 ? static_cast<float>(st[0] / static_cast<double>(nv)) : 0.f;
    a.inv_nvalid[k] = nv > 0 ? static_cast<float>(1.0 / static_cast<double>(nv)) : 0.f;
    if (a.dtau) a.dtau[k] = nv > 0 ? static_cast<float>(stt[0] / static_cast<double>(nv)) : 0.f;
  }
}

// ---- dL/dz in place: G = tau (softmax - onehot) / Nvalid --------------------
// The buffer holds p~ = bf16(exp(z - m_t)) for the column tile t of each
// entry, so softmax = p~ * exp(m_t - lse).  The target entry is recomputed
// as expm1(-(lse - z_y)), from the lse - z_y that the log-sum-exp pass forms
// without cancellation, so that p_y - 1 keeps its relative precision.

// End of the rows past the kept ones that the dW product may read: its
// reduction covers the final module's kept rows in whole 128-row blocks (its
// N rows, rounded, when it keeps none), so those rows are zeroed.
__device__ __forceinline__ int64_t dw_zero_end(const RowArgs& a, int64_t M) {
  const int64_t fin0 = a.offsets[a.K - 1];
  const int64_t kept = a.offsets[a.K] - fin0;
  const int64_t span = kept > 0 ? kept : a.N;
  return min(M, fin0 + (span + 127) / 128 * 128);
}

// The gradient pass without bias gradients, in two launches.
// grad_classify_kernel: 32 rows per CTA.  One coalesced look at the rows decides
// what each needs: the whole row (a kept row without a per-row factor: P
// becomes G; a masked row without compaction), listed for grad_rows_kernel;
// its target entry and x̂ row only (a final-module row with a factor: dW =
// G^T x̂ = P'^T (c x̂)), done here by one warp; or nothing (an auxiliary row with
// a factor: the dX̂ epilogue forms its gradient).  kGradZeroCtas more CTAs zero
// the rows past the kept ones that dW reads, one row at a time each.
constexpr int kGradRowsPerCta = 32;
constexpr int kGradZeroCtas = 128;

__global__ void __launch_bounds__(256) grad_classify_kernel(const RowArgs a) {
  __shared__ int s_rows[kGradRowsPerCta];
  __shared__ int s_count;
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const int64_t row_base = static_cast<int64_t>(blockIdx.x) * kGradRowsPerCta;
  const bool compact = a.kept_local != nullptr;
  const int64_t nchk = (M + kGradRowsPerCta - 1) / kGradRowsPerCta;
  if (blockIdx.x >= nchk) {
    if (!compact) return;
    const int64_t zend = dw_zero_end(a, M);
    const int nvec = a.ldp / 8;
    for (int64_t row = a.offsets[a.K] + (blockIdx.x - nchk); row < zend; row += kGradZeroCtas) {
      uint4* P = reinterpret_cast<uint4*>(a.P + row * a.ldp);
      for (int v = threadIdx.x; v < nvec; v += 256) P[v] = make_uint4(0, 0, 0, 0);
    }
    return;
  }
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    const int64_t row = row_base + lane;
    const int64_t mk = compact ? a.offsets[a.K] : M;
    const int64_t fin0 = compact ? a.offsets[a.K - 1] : static_cast<int64_t>(a.K - 1) * a.N;
    int kind = 0;                 // 1: the whole row, 2: target entry and x̂ row
    if (row < mk) {
      const bool factor = a.row_fa != nullptr && a.row_fa[row] >= 0.f;
      kind = !factor ? 1 : row >= fin0 ? 2 : 0;
    }
    const unsigned below = (1u << lane) - 1u;
    const unsigned whole = __ballot_sync(0xffffffffu, kind == 1);
    int base = 0;
    if (lane == 0 && whole != 0u) base = atomicAdd(a.grad_count, __popc(whole));
    base = __shfl_sync(0xffffffffu, base, 0);
    if (kind == 1 && in_bounds(base + __popc(whole & below) < M, a.flags))
      a.grad_list[base + __popc(whole & below)] = static_cast<int32_t>(row);
    const unsigned part = __ballot_sync(0xffffffffu, kind == 2);
    if (kind == 2) s_rows[__popc(part & below)] = lane;
    if (lane == 0) s_count = __popc(part);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < s_count; i += 8) {
    const int64_t rk = row_base + s_rows[i];
    const int64_t tk = compact ? a.orig_row[rk] : rk;
    const int kf = static_cast<int>(tk / a.N);
    const int yf = compact ? a.tgt_c[rk] : a.targets[rk];
    const float tauf = a.tau ? a.tau[kf] : 1.f;
    const float c = tauf * a.inv_nvalid[kf] * a.row_fa[rk];
    if (lane == 0 && in_bounds(yf >= 0 && yf < a.V, a.flags))
      a.P[rk * a.ldp + yf] = __bfloat16_as_ushort(__float2bfloat16(expm1f(-a.nll[rk]) * expf(a.lse[rk])));
    uint4* xr = reinterpret_cast<uint4*>(a.xhat + rk * a.d);
    for (int v = lane; v < a.d / 8; v += 32) {
      float f[8];
      unpack8(xr[v], f);
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] *= c;
      xr[v] = make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
    }
  }
}

// grad_rows_kernel: the listed rows, one per CTA at a time (a grid of a few CTAs
// per SM walks the list), contiguous 16-byte vectors across the row.
__global__ void __launch_bounds__(256) grad_rows_kernel(const RowArgs a) {
  extern __shared__ float ctile[];
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const bool compact = a.kept_local != nullptr;
  const int nvec = a.ldp / 8;
  const int count = *a.grad_count;
  if (!in_bounds(count <= M, a.flags)) return;
  for (int i = blockIdx.x; i < count; i += gridDim.x) {
    const int64_t row = a.grad_list[i];
    if (!in_bounds(row >= 0 && row < M, a.flags)) continue;    // uniform across the CTA
    uint4* P = reinterpret_cast<uint4*>(a.P + row * a.ldp);
    const int64_t tok = compact ? a.orig_row[row] : row;
    const int k = static_cast<int>(tok / a.N);
    const int y = compact ? a.tgt_c[row] : a.targets[row];
    if (!compact && !token_kept(a, row, y)) {
      for (int v = threadIdx.x; v < nvec; v += 256) P[v] = make_uint4(0, 0, 0, 0);
      continue;                   // uniform across the CTA
    }
    const float tau = a.tau ? a.tau[k] : 1.f;
    const float w = a.inv_nvalid[k] * tau;
    const float l = a.lse[row];
    __syncthreads();              // the previous row's factors are no longer read
    for (int t = threadIdx.x; t < a.n_tiles_v; t += 256)
      ctile[t] = expf(a.stats[static_cast<int64_t>(t) * M + row].x - l) * w;
    const float gy = expm1f(-a.nll[row]) * w;    // p_y - 1 at full relative precision
    __syncthreads();
    constexpr int kAhead = 4;                     // vectors in flight per thread
    for (int vb = threadIdx.x; vb < nvec; vb += 256 * kAhead) {
      uint4 in[kAhead];
#pragma unroll
      for (int u = 0; u < kAhead; ++u) {
        const int v = vb + 256 * u;
        if (v < nvec && v * 8 < a.V) in[u] = P[v];
      }
#pragma unroll
      for (int u = 0; u < kAhead; ++u) {
        const int v = vb + 256 * u;
        if (v >= nvec) break;
        const int v0 = v * 8;
        if (v0 >= a.V) {
          P[v] = make_uint4(0, 0, 0, 0);
          continue;
        }
        if (!in_bounds(v0 / kBN < a.n_tiles_v, a.flags)) continue;
        const float c = ctile[v0 / kBN];
        float f[8];
        unpack8(in[u], f);
#pragma unroll
        for (int j = 0; j < 8; ++j) f[j] *= c;
        if (v0 + 8 > a.V) {          // the vector that crosses V
#pragma unroll
          for (int j = 0; j < 8; ++j) f[j] = v0 + j < a.V ? f[j] : 0.f;
        }
        const int ycol = y - v0;
        if (static_cast<unsigned>(ycol) < 8u) {   // the vector holding the target
#pragma unroll
          for (int j = 0; j < 8; ++j) f[j] = j == ycol ? gy : f[j];
        }
        P[v] = make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
      }
    }
  }
}

// With the bias gradient: a CTA owns kGradRows rows of one module and 2048
// columns (8 tiles), each thread one 8-column vector down those rows, so it
// also sums dL/dz over its rows (fixed order, per row chunk).  Rows whose
// gradient is P times a per-row factor (row_fa >= 0) are summed the same way
// but keep their exponentials in P: the dX̂ epilogue applies the factor to an
// auxiliary row, and a final-module row gets its target entry and its x̂ row
// scaled, as in the pass without bias gradients.
__global__ void __launch_bounds__(256, 4) grad_colsum_kernel(const RowArgs a) {
  __shared__ float cfac[kGradRows][8];     // exp(m_t - lse) / Nvalid per row and tile
  // per row, read together: the target (-1: masked or zero row), (p_y - 1) /
  // Nvalid, the x̂ scale of a final-module factor row (else NaN), and 1 when P
  // keeps the row's exponentials
  __shared__ float4 srow[kGradRows];
  __shared__ unsigned short sty[kGradRows];    // a final-module factor row's target entry
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  // one-dimensional grid, the 2048-column slice fastest (the CTAs running
  // together read whole rows): blockIdx.x = (module, row chunk) * slices + slice
  const int nslice = (a.ldp / 8 + 255) / 256;
  const int slice = static_cast<int>(blockIdx.x % static_cast<unsigned>(nslice));
  const int unit = static_cast<int>(blockIdx.x / static_cast<unsigned>(nslice));
  const int k = unit / a.db_chunks;
  const int chunk = unit - k * a.db_chunks;
  // compacted: module k's kept tokens are rows [offsets[k], offsets[k + 1]); the
  // final module's chunks also zero the rows past Mk that the dW product may
  // read (their contents are stale: written as zeros, never scaled)
  const bool compact = a.kept_local != nullptr;
  const int64_t mbase = compact ? a.offsets[k] : static_cast<int64_t>(k) * a.N;
  const int64_t mkept = compact ? a.offsets[k + 1] : mbase + a.N;
  const int64_t row0 = mbase + static_cast<int64_t>(chunk) * kGradRows;
  const int64_t end = (compact && k < a.K - 1) ? mkept : compact ? dw_zero_end(a, M) : mbase + a.N;
  const int rows = row0 >= end ? 0 : static_cast<int>(end - row0 < kGradRows ? end - row0 : kGradRows);
  const int t0 = slice * 8;                      // first 256-column tile of this CTA
  if (!in_bounds(k < a.K && row0 + rows <= M, a.flags)) return;
  const float w = a.inv_nvalid[k];
  const float tau = a.tau ? a.tau[k] : 1.f;
  if (threadIdx.x < rows) {
    const int r = threadIdx.x;
    const int64_t i = row0 + r;
    const int y = compact ? (i < mkept ? a.tgt_c[i] : -1) : a.targets[i];
    const bool kept = compact ? i < mkept : token_kept(a, i, y);
    const float l = a.lse[i];
    const float wr = kept ? w : 0.f;
#pragma unroll
    for (int tt = 0; tt < 8; ++tt) {
      const int t = t0 + tt;
      cfac[r][tt] = (wr != 0.f && t < a.n_tiles_v)
                        ? expf(a.stats[static_cast<int64_t>(t) * M + i].x - l) * wr : 0.f;
    }
    const bool factor = kept && a.row_fa != nullptr && a.row_fa[i] >= 0.f;
    const bool fin = factor && k == a.K - 1;
    srow[r] = make_float4(__int_as_float(kept ? y : -1), kept ? expm1f(-a.nll[i]) * wr : 0.f,
                          fin ? tau * w * a.row_fa[i] : __int_as_float(0x7fc00000),
                          __int_as_float(factor ? 1 : 0));
    sty[r] = fin ? __bfloat16_as_ushort(__float2bfloat16(expm1f(-a.nll[i]) * expf(l))) : 0;
  }
  __syncthreads();
  if (k == a.K - 1 && a.row_fa != nullptr) {
    // x̂ rows of the final module's factor rows times tau/Nvalid e^{-lse}
    // (G^T x̂ = P'^T (c x̂)); the CTAs of a row chunk share each row's vectors
    const int nvd = a.d / 8;
    const int v0 = static_cast<int>(static_cast<int64_t>(slice) * nvd / nslice);
    const int len = static_cast<int>(static_cast<int64_t>(slice + 1) * nvd / nslice) - v0;
    for (int idx = threadIdx.x; len > 0 && idx < rows * len; idx += 256) {
      const int r = idx / len;
      const float c = srow[r].z;
      if (c != c) continue;
      uint4* xr = reinterpret_cast<uint4*>(a.xhat + (row0 + r) * a.d) + v0 + (idx - r * len);
      float f[8];
      unpack8(*xr, f);
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] *= c;
      *xr = make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
    }
  }
  const int vec = slice * 256 + threadIdx.x;         // 8-column vector of this thread
  if (vec * 8 >= a.ldp) return;
  const int col0 = vec * 8;
  const int tt = threadIdx.x >> 5;                    // 32 vectors = one 256-column tile
  float colsum[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) colsum[j] = 0.f;
  uint4* P = reinterpret_cast<uint4*>(a.P + row0 * a.ldp) + vec;
  const int64_t stride = a.ldp / 8;
  constexpr int kAhead = 8;                           // rows in flight per thread
  const bool vfull = col0 + 8 <= a.V;                 // every column of the vector in V
  for (int r0 = 0; r0 < rows; r0 += kAhead) {
    uint4 in[kAhead];
#pragma unroll
    for (int u = 0; u < kAhead; ++u)
      if (r0 + u < rows) in[u] = P[(r0 + u) * stride];
#pragma unroll
    for (int u = 0; u < kAhead; ++u) {
      const int r = r0 + u;
      if (r >= rows) break;
      const float4 rd = srow[r];
      const int yr = __float_as_int(rd.x);
      if (yr < 0) {                 // a masked or zero row (warp-uniform): G = 0
        P[r * stride] = make_uint4(0, 0, 0, 0);
        continue;
      }
      const float c = cfac[r][tt];
      const int ycol = yr - col0;
      float g[8];
      unpack8(in[u], g);
#pragma unroll
      for (int j = 0; j < 8; ++j) g[j] *= c;
      if (static_cast<unsigned>(ycol) < 8u) {      // the thread holding the target
        const float gy = rd.y;
#pragma unroll
        for (int j = 0; j < 8; ++j) g[j] = j == ycol ? gy : g[j];
      }
      if (!vfull) {                 // the vector that crosses V
#pragma unroll
        for (int j = 0; j < 8; ++j) g[j] = col0 + j < a.V ? g[j] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) colsum[j] += g[j];
      if (__float_as_int(rd.w) == 0) {
        P[r * stride] = make_uint4(pack2(g[0] * tau, g[1] * tau), pack2(g[2] * tau, g[3] * tau),
                                   pack2(g[4] * tau, g[5] * tau), pack2(g[6] * tau, g[7] * tau));
      } else if (static_cast<unsigned>(ycol) < 8u && rd.z == rd.z) {
        // a final-module factor row: its target entry becomes (p_y - 1) e^{lse}
        reinterpret_cast<unsigned short*>(P + r * stride)[ycol] = sty[r];
      }
    }
  }
  if (!in_bounds(chunk < a.db_chunks && col0 + 8 <= a.ldp, a.flags)) return;
  float* out = a.db_part + (static_cast<int64_t>(k) * a.db_chunks + chunk) * a.ldp + col0;
  reinterpret_cast<float4*>(out)[0] = make_float4(colsum[0], colsum[1], colsum[2], colsum[3]);
  reinterpret_cast<float4*>(out)[1] = make_float4(colsum[4], colsum[5], colsum[6], colsum[7]);
}

// db_k[v] = sum over the row chunks of module k (fixed order)
__global__ void __launch_bounds__(256) dbias_reduce_kernel(const RowArgs a) {
  const int k = blockIdx.y;
  const int v = blockIdx.x * 256 + threadIdx.x;
  if (v >= a.V) return;
  float acc = 0.f;
  for (int c = 0; c < a.db_chunks; ++c)
    acc += a.db_part[(static_cast<int64_t>(k) * a.db_chunks + c) * a.ldp + v];
  a.dbias[static_cast<int64_t>(k) * a.V + v] = acc;
}

// ---- dgamma of the final module: the fixed-order sum of the partial sums per
// 32-row block that the RMSNorm backward (fused into the dX̂ GEMM) wrote -----

// One CTA per 32 columns: warp w sums a fixed segment of the partial rows for
// its 32 columns (lane = column, 128-byte rows), then warp 0 adds the eight
// segment sums in order.
__global__ void __launch_bounds__(256) dgamma_reduce_kernel(const RowArgs a) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int j = blockIdx.x * 32 + lane;
  // compacted: the final module's kept tokens are rows [offsets[K-1], Mk), so
  // the 32-row blocks holding them are fewer than for all its tokens
  int chunks = a.dg_chunks;
  if (a.kept_local != nullptr) {
    const int64_t f0 = a.offsets[a.K - 1], f1 = a.offsets[a.K];
    chunks = f1 > f0 ? static_cast<int>(((f1 - 1) >> 5) - (f0 >> 5) + 1) : 0;
    chunks = min(chunks, a.dg_chunks);
  }
  const int seg = (chunks + 7) / 8;
  const int c1 = min(chunks, (warp + 1) * seg);
  float acc = 0.f;
  if (j < a.d) {
    int c = warp * seg;
    for (; c + 8 <= c1; c += 8) {          // eight loads in flight, added in order
      float x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = a.dgamma_part[static_cast<int64_t>(c + u) * a.d + j];
#pragma unroll
      for (int u = 0; u < 8; ++u) acc += x[u];
    }
    for (; c < c1; ++c) acc += a.dgamma_part[static_cast<int64_t>(c) * a.d + j];
  }
  __shared__ float seg_sum[8][32];
  seg_sum[warp][lane] = acc;
  __syncthreads();
  if (warp == 0 && j < a.d) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += seg_sum[w][lane];
    a.dgamma[j] = t;
  }
}

}  // namespace

// Smallest register cache (vectors per lane) that holds a row of d elements;
// 0 (re-read the row) above d = 2048, where a larger cache costs more in
// occupancy than the second read from L2 (measured at d = 2560).
static int vectors_per_lane(int d) {
  const int v = (d / 8 + 31) / 32;
  return v <= 1 ? 1 : v <= 2 ? 2 : v <= 4 ? 4 : v <= 8 ? 8 : 0;
}

cudaError_t launch_rmsnorm_fwd(const RowArgs& a, cudaStream_t s) {
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const unsigned grid = static_cast<unsigned>((M + 7) / 8);
  switch (vectors_per_lane(a.d)) {
    case 1: rmsnorm_fwd_kernel<1><<<grid, 256, 0, s>>>(a); break;
    case 2: rmsnorm_fwd_kernel<2><<<grid, 256, 0, s>>>(a); break;
    case 4: rmsnorm_fwd_kernel<4><<<grid, 256, 0, s>>>(a); break;
    case 8: rmsnorm_fwd_kernel<8><<<grid, 256, 0, s>>>(a); break;
    default: rmsnorm_fwd_kernel<0><<<grid, 256, 0, s>>>(a); break;
  }
  return launched();
}

cudaError_t launch_keep_scan(const RowArgs& a, cudaStream_t s) {
  keep_scan_kernel<<<dim3(a.nchunks, a.K), kScanRows, 0, s>>>(a);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  keep_offsets_kernel<<<1, 1024, 0, s>>>(a);
  return launched();
}

cudaError_t launch_lse(const RowArgs& a, cudaStream_t s, bool heads) {
  if (heads)
    lse_kernel<kLseHeads><<<dim3(a.part_blocks, a.K), 256, 0, s>>>(a);
  else
    lse_kernel<kLseTrain><<<dim3(a.part_blocks, a.K), 256, 0, s>>>(a);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  module_mean_kernel<<<a.K, 256, 0, s>>>(a);
  return launched();
}

cudaError_t launch_exit_lse(const RowArgs& a, cudaStream_t s) {
  lse_kernel<kLseExit><<<dim3(a.part_blocks, a.K), 256, 0, s>>>(a);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  module_mean_kernel<<<a.K, 256, 0, s>>>(a);
  return launched();
}

cudaError_t launch_grad(const RowArgs& a, cudaStream_t s) {
  if (a.dbias) {
    const int64_t ctas = static_cast<int64_t>(a.K) * a.db_chunks * ((a.ldp / 8 + 255) / 256);
    grad_colsum_kernel<<<static_cast<unsigned>(ctas), 256, 0, s>>>(a);
    cudaError_t e = launched();
    if (e != cudaSuccess) return e;
    dbias_reduce_kernel<<<dim3((a.V + 255) / 256, a.K), 256, 0, s>>>(a);
    return launched();
  }
  const int64_t M = static_cast<int64_t>(a.K) * a.N;
  const size_t smem = static_cast<size_t>(a.n_tiles_v) * sizeof(float);
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(grad_rows_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  const int64_t ctas = (M + kGradRowsPerCta - 1) / kGradRowsPerCta + kGradZeroCtas;
  grad_classify_kernel<<<static_cast<unsigned>(ctas), 256, 0, s>>>(a);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  grad_rows_kernel<<<static_cast<unsigned>(a.grad_ctas > 0 ? a.grad_ctas : 1), 256, smem, s>>>(a);
  return launched();
}

cudaError_t launch_dgamma_reduce(const RowArgs& a, cudaStream_t s) {
  dgamma_reduce_kernel<<<(a.d + 31) / 32, 256, 0, s>>>(a);
  return launched();
}

}  // namespace solo
