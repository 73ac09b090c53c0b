// Host side of the C ABI: argument checks, workspace layout, TMA tensor maps
// and the launch sequence of one call.
//
// Launch sequence (all on the caller's stream, no host synchronisation):
//   rmsnorm      r_i and xhat = bf16(gamma h r)                  [K*N, d]
//   logits       tensor-core xhat W^T; per (row, 256-column tile) max and
//                sum of exp, target logit, bf16 exp(z - tile max)  [K*N, V]
//   lse          log-sum-exp per row, token loss, module means, 1/Nvalid
//   grad         (softmax - onehot)/Nvalid in place, bf16        [K*N, V]
//   dxhat        tensor-core G W with the RMSNorm backward in its epilogue:
//                bf16 dH and the final module's dgamma partial sums [K*N, d]
//   norm_bwd     the same for the tiles whose last wave was cut along V
//                (their fp32 parts summed first, from the partial-tile slots)
//   dW           tensor-core G^T xhat over the final module       [V, d]
//   dgamma       fixed-order sum of the partials                  [d]
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "../../include/solo_readout.h"
#include "internal.h"

namespace solo {

namespace {
std::atomic<uint64_t> g_launches{0};
}  // namespace

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
uint64_t launch_count() { return g_launches.load(std::memory_order_relaxed); }

}  // namespace solo

namespace {

using namespace solo;

constexpr size_t kAlign = 1024;
// Largest vocabulary: the gradient pass keeps one float per 256-column tile of
// a row in shared memory (128 KB at this size).
constexpr int32_t kMaxVocab = 1 << 23;
// Tile raster (in 256-row pair blocks) per product, from a sweep on GB300.
constexpr int kGroupLogits = 16;
constexpr int kGroupDxhat = 4;
constexpr int kGroupDW = 4;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Layout {
  int64_t M = 0;
  int ldp = 0;
  int n_tiles_v = 0;
  int part_blocks = 0;
  int dg_chunks = 0;
  int db_chunks = 0;
  size_t flags = 0, r = 0, lse = 0, zy = 0, edz = 0, nll = 0, part_sum = 0, part_cnt = 0;
  size_t inv_nvalid = 0;
  size_t stats = 0, xhat = 0, P = 0, dgp = 0;
  size_t usum = 0, sy = 0, part_tau = 0, db_part = 0, aux = 0, total = 0;
  size_t kept_local = 0, chunk_base = 0, offsets = 0, orig_row = 0, tgt_c = 0;
  size_t grad_list = 0, grad_count = 0;
  size_t row_fa = 0, row_fb = 0;
  int aux_slots = 0;
  int nchunks = 0;
};

solo_status_t check_dims(const solo_dims_t* d) {
  if (d == nullptr) return SOLO_ERR_INVALID_ARG;
  if (d->K < 1 || d->K > SOLO_MAX_MODULES) return SOLO_ERR_INVALID_ARG;
  if (d->N < 1 || d->d < 8 || d->V < 1) return SOLO_ERR_INVALID_ARG;
  if (!(d->eps >= 0.0f) || !std::isfinite(d->eps)) return SOLO_ERR_INVALID_ARG;
  if (d->d % 8 != 0) return SOLO_ERR_UNSUPPORTED_SHAPE;
  // row and column coordinates of the tensor-core operands are 32-bit
  const int64_t M = static_cast<int64_t>(d->K) * d->N;
  if (M > (int64_t{1} << 31) - 1 - kBM) return SOLO_ERR_UNSUPPORTED_SHAPE;
  if (d->V > kMaxVocab || d->d > (1 << 20)) return SOLO_ERR_UNSUPPORTED_SHAPE;
  // tile counts of the products are 32-bit
  const int64_t row_blocks = (M + 2 * kBM - 1) / (2 * kBM);
  const int64_t col_blocks = (static_cast<int64_t>(d->V) + kBN - 1) / kBN;
  if (row_blocks * col_blocks > (int64_t{1} << 31) - 1) return SOLO_ERR_UNSUPPORTED_SHAPE;
  return SOLO_OK;
}

Layout make_layout(const solo_dims_t& d) {
  Layout L;
  L.M = static_cast<int64_t>(d.K) * d.N;
  L.ldp = static_cast<int>(align_up(d.V, 8));
  L.n_tiles_v = (d.V + kBN - 1) / kBN;
  L.part_blocks = static_cast<int>((d.N + 255) / 256);
  // dgamma partial sums per 32-row block holding rows of the final module: its
  // kept tokens start at any compact row, so they span at most N/32 + 1 blocks
  L.dg_chunks = static_cast<int>((d.N + 31) / 32 + 1);
  L.db_chunks = static_cast<int>((d.N + kGradRows - 1) / kGradRows);
  const size_t M = static_cast<size_t>(L.M);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, kAlign);
    return at;
  };
  L.flags = take(256);
  L.r = take(M * 4);
  L.lse = take(M * 4);
  L.zy = take(M * 4);
  L.edz = take(M * 4);
  L.nll = take(M * 4);
  L.part_sum = take(static_cast<size_t>(d.K) * L.part_blocks * 8);
  L.part_cnt = take(static_cast<size_t>(d.K) * L.part_blocks * 4);
  L.inv_nvalid = take(SOLO_MAX_MODULES * 4);
  L.stats = take(static_cast<size_t>(L.n_tiles_v) * M * 8);
  L.xhat = take(M * d.d * 2);
  L.P = take(M * static_cast<size_t>(L.ldp) * 2);
  L.dgp = take(static_cast<size_t>(L.dg_chunks) * d.d * 4);
  // heads' temperature and bias gradients
  L.usum = take(static_cast<size_t>(L.n_tiles_v) * M * 4);
  L.sy = take(M * 4);
  L.part_tau = take(static_cast<size_t>(d.K) * L.part_blocks * 8);
  L.db_part = take(static_cast<size_t>(d.K) * L.db_chunks * L.ldp * 4);
  // partial tiles of the dX̂ and dW products' last wave (one product at a
  // time; every part of a cut dX̂ tile, parts 1.. of a cut dW tile)
  const int64_t nb = (d.d + kBN - 1) / kBN;
  const int64_t tiles_dx = (L.M + 2 * kBM - 1) / (2 * kBM) * nb;
  const int64_t tiles_dw = (d.V + 2 * kBM - 1) / (2 * kBM) * nb;
  L.aux_slots = std::max(split_aux_slots(tiles_dx, (d.V + kBK - 1) / kBK, true),
                         split_aux_slots(tiles_dw, (d.N + kBK - 1) / kBK, false));
  L.aux = take(static_cast<size_t>(std::max(L.aux_slots, 1)) * 2 * kBM * kBN * 4);
  // kept-token compaction: in-chunk ranks, chunk prefixes, module offsets, the
  // token and target of every compact row
  L.nchunks = static_cast<int>((d.N + kScanRows - 1) / kScanRows);
  L.kept_local = take(M * 4);
  L.chunk_base = take(static_cast<size_t>(d.K) * L.nchunks * 4);
  L.offsets = take((SOLO_MAX_MODULES + 1) * 4);
  L.orig_row = take(M * 4);
  L.tgt_c = take(M * 4);
  // per-row factors of the rows whose gradient the dX̂ epilogue forms
  L.row_fa = take(M * 4);
  L.row_fb = take(M * 4);
  // rows whose gradient pass takes the whole row, and their count
  L.grad_list = take(M * 4);
  L.grad_count = take(4);
  L.total = off;
  return L;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Byte ranges of a call's buffers: an output (or the workspace) may overlap
// no other buffer; inputs may share memory with each other (they are only
// read).
struct Ranges {
  static constexpr int kMax = 2 * SOLO_MAX_MODULES + 16;
  uintptr_t lo[kMax];
  uintptr_t hi[kMax];
  bool out[kMax];
  int n = 0;
  void add(const void* p, size_t bytes, bool is_out) {
    if (p == nullptr || bytes == 0 || n == kMax) return;
    lo[n] = reinterpret_cast<uintptr_t>(p);
    hi[n] = lo[n] + bytes;
    out[n] = is_out;
    ++n;
  }
  bool any_output_overlap() const {
    for (int i = 0; i < n; ++i)
      for (int j = i + 1; j < n; ++j)
        if ((out[i] || out[j]) && lo[i] < hi[j] && lo[j] < hi[i]) return true;
    return false;
  }
};

// ---- per-device setup ------------------------------------------------------------

struct DeviceInfo {
  bool ready = false;
  bool sm103 = false;
  int sms = 0;
};

std::mutex g_dev_mu;
DeviceInfo g_dev[64];

solo_status_t device_setup(int* sms, int* device = nullptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SOLO_ERR_CUDA;
  if (dev < 0 || dev >= 64) return SOLO_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_dev_mu);
  DeviceInfo& info = g_dev[dev];
  if (!info.ready) {
    int major = 0, minor = 0, sms_ = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms_, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return SOLO_ERR_CUDA;
    info.sm103 = (major == 10 && minor == 3);
    info.sms = sms_;
    if (info.sm103 && (gemm_prepare(dev) != cudaSuccess || flash_prepare(dev) != cudaSuccess))
      return SOLO_ERR_CUDA;
    info.ready = true;
  }
  if (!info.sm103) return SOLO_ERR_NOT_SM103;
  *sms = info.sms;
  if (device) *device = dev;
  return SOLO_OK;
}

// ---- TMA tensor maps ----------------------------------------------------------------

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D row-major tensor [outer, inner] with a row pitch of row_bytes, loaded
// or stored in boxes of [box_outer, box_inner] with 128-byte swizzle; reads
// outside the tensor return zeros and writes outside it are dropped.
bool make_map(CUtensorMap* m, CUtensorMapDataType dt, const void* ptr, uint64_t inner,
              uint64_t outer, uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

solo_status_t run(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                  const solo_bf16_t* gamma, const solo_bf16_t* W, const int32_t* targets,
                  const uint8_t* mask, const solo_heads_t* heads, float* loss_tok,
                  float* loss_mean, solo_bf16_t* const* dhidden, float* dW, float* dgamma,
                  void* workspace, size_t workspace_bytes, cudaStream_t stream,
                  void* const* events, int32_t n_events, bool clear_flags = true) {
  // -------- host-side checks: nothing is enqueued when one fails
  solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  const solo_dims_t& D = *dims;
  if (hidden == nullptr || dhidden == nullptr || gamma == nullptr || W == nullptr ||
      targets == nullptr || loss_mean == nullptr || workspace == nullptr)
    return SOLO_ERR_INVALID_ARG;
  if (events != nullptr && n_events != SOLO_NUM_STAGES + 1) return SOLO_ERR_INVALID_ARG;
  for (int k = 0; k < D.K; ++k) {
    if (hidden[k] == nullptr || dhidden[k] == nullptr) return SOLO_ERR_INVALID_ARG;
    if (!aligned16(hidden[k]) || !aligned16(dhidden[k])) return SOLO_ERR_MISALIGNED;
  }
  if (!aligned16(gamma) || !aligned16(W) || !aligned16(workspace) ||
      (reinterpret_cast<uintptr_t>(targets) & 3u) || (dW && !aligned16(dW)) ||
      (dgamma && (reinterpret_cast<uintptr_t>(dgamma) & 3u)) ||
      (loss_tok && (reinterpret_cast<uintptr_t>(loss_tok) & 3u)) ||
      (reinterpret_cast<uintptr_t>(loss_mean) & 3u))
    return SOLO_ERR_MISALIGNED;
  const float* tau = heads ? heads->tau : nullptr;
  const float* bias = heads ? heads->bias : nullptr;
  float* dtau = heads ? heads->dtau : nullptr;
  float* dbias = heads ? heads->dbias : nullptr;
  if ((reinterpret_cast<uintptr_t>(tau) & 3u) || (reinterpret_cast<uintptr_t>(bias) & 3u) ||
      (reinterpret_cast<uintptr_t>(dtau) & 3u) || (reinterpret_cast<uintptr_t>(dbias) & 3u))
    return SOLO_ERR_MISALIGNED;
  const bool affine = tau || bias || dtau;   // z = tau s + b (and its temperature gradient)
  const Layout L = make_layout(D);
  if (workspace_bytes < L.total) return SOLO_ERR_WORKSPACE_TOO_SMALL;
  {
    const size_t K = static_cast<size_t>(D.K), N = static_cast<size_t>(D.N);
    const size_t dd = static_cast<size_t>(D.d), VV = static_cast<size_t>(D.V);
    Ranges rg;
    for (int k = 0; k < D.K; ++k) {
      rg.add(hidden[k], N * dd * 2, false);
      rg.add(dhidden[k], N * dd * 2, true);
    }
    rg.add(gamma, dd * 2, false);
    rg.add(W, VV * dd * 2, false);
    rg.add(targets, K * N * 4, false);
    rg.add(mask, K * N, false);
    rg.add(tau, K * 4, false);
    rg.add(bias, K * VV * 4, false);
    rg.add(loss_tok, K * N * 4, true);
    rg.add(loss_mean, K * 4, true);
    rg.add(dW, VV * dd * 4, true);
    rg.add(dgamma, dd * 4, true);
    rg.add(dtau, K * 4, true);
    rg.add(dbias, K * VV * 4, true);
    rg.add(workspace, L.total, true);
    if (rg.any_output_overlap()) return SOLO_ERR_INVALID_ARG;
  }

  // -------- device
  int sms = 0;
  st = device_setup(&sms);
  if (st != SOLO_OK) return st;

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  RowArgs ra;
  std::memset(&ra, 0, sizeof(ra));
  for (int k = 0; k < D.K; ++k) {
    ra.hidden[k] = hidden[k];
    ra.dhidden[k] = dhidden[k];
  }
  ra.N = D.N;
  ra.K = D.K;
  ra.d = D.d;
  ra.V = D.V;
  ra.ldp = L.ldp;
  ra.n_tiles_v = L.n_tiles_v;
  ra.ignore_index = D.ignore_index;
  ra.eps = D.eps;
  ra.gamma = gamma;
  ra.targets = targets;
  ra.mask = mask;
  ra.r = reinterpret_cast<float*>(ws + L.r);
  ra.xhat = reinterpret_cast<uint16_t*>(ws + L.xhat);
  ra.lse = reinterpret_cast<float*>(ws + L.lse);
  ra.zy = reinterpret_cast<float*>(ws + L.zy);
  ra.edz = reinterpret_cast<float*>(ws + L.edz);
  ra.nll = reinterpret_cast<float*>(ws + L.nll);
  ra.stats = reinterpret_cast<float2*>(ws + L.stats);
  ra.part_sum = reinterpret_cast<double*>(ws + L.part_sum);
  ra.part_cnt = reinterpret_cast<int32_t*>(ws + L.part_cnt);
  ra.part_blocks = L.part_blocks;
  ra.inv_nvalid = reinterpret_cast<float*>(ws + L.inv_nvalid);
  ra.loss_tok = loss_tok;
  ra.loss_mean = loss_mean;
  ra.P = reinterpret_cast<uint16_t*>(ws + L.P);
  ra.dgamma_part = reinterpret_cast<float*>(ws + L.dgp);
  ra.dg_chunks = L.dg_chunks;
  ra.dgamma = dgamma;
  ra.flags = reinterpret_cast<uint32_t*>(ws + L.flags);
  ra.tau = tau;
  ra.usum = reinterpret_cast<float*>(ws + L.usum);
  ra.sy = reinterpret_cast<float*>(ws + L.sy);
  ra.part_tau = reinterpret_cast<double*>(ws + L.part_tau);
  ra.dtau = dtau;
  ra.dbias = dbias;
  ra.db_part = reinterpret_cast<float*>(ws + L.db_part);
  ra.db_chunks = L.db_chunks;
  // masked tokens are skipped: the kept ones are compacted into rows [0, Mk)
  ra.kept_local = reinterpret_cast<int32_t*>(ws + L.kept_local);
  ra.chunk_base = reinterpret_cast<int32_t*>(ws + L.chunk_base);
  ra.nchunks = L.nchunks;
  ra.offsets = reinterpret_cast<int32_t*>(ws + L.offsets);
  ra.orig_row = reinterpret_cast<int32_t*>(ws + L.orig_row);
  ra.tgt_c = reinterpret_cast<int32_t*>(ws + L.tgt_c);
  // gradients formed from the stored exponentials and per-row factors where
  // they allow it: in the dX̂ epilogue (auxiliary rows), from a target entry and
  // a scaled x̂ row (final-module rows)
  ra.row_fa = reinterpret_cast<float*>(ws + L.row_fa);
  ra.row_fb = reinterpret_cast<float*>(ws + L.row_fb);
  ra.grad_list = reinterpret_cast<int32_t*>(ws + L.grad_list);
  ra.grad_count = reinterpret_cast<int32_t*>(ws + L.grad_count);
  ra.grad_ctas = 4 * sms;

  const uint64_t M = static_cast<uint64_t>(L.M);
  const uint64_t d = static_cast<uint64_t>(D.d);
  const uint64_t V = static_cast<uint64_t>(D.V);
  const auto BF = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const auto F32 = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  CUtensorMap mX_k, mW_k, mP_st, mG_k, mW_mn, mG_mn, mX_mn, mDW, mAux;
  float* aux = reinterpret_cast<float*>(ws + L.aux);
  bool ok = make_map(&mX_k, BF, ra.xhat, d, M, d * 2, 64, kBM) &&
            make_map(&mAux, F32, aux, kBN,
                     static_cast<uint64_t>(std::max(L.aux_slots, 1)) * 2 * kBM, kBN * 4, 32,
                     32) &&
            make_map(&mW_k, BF, W, d, V, d * 2, 64, kBN / 2) &&
            make_map(&mP_st, BF, ra.P, V, M, static_cast<uint64_t>(L.ldp) * 2, 64, 32) &&
            make_map(&mG_k, BF, ra.P, V, M, static_cast<uint64_t>(L.ldp) * 2, 64, kBM) &&
            make_map(&mW_mn, BF, W, d, V, d * 2, 64, kBK);
  if (ok && dW) {
    ok = make_map(&mG_mn, BF, ra.P, V, M, static_cast<uint64_t>(L.ldp) * 2, 64, kBK) &&
         make_map(&mX_mn, BF, ra.xhat, d, M, d * 2, 64, kBK) &&
         make_map(&mDW, F32, dW, d, V, d * 4, 32, 32);
  }
  if (!ok) return SOLO_ERR_CUDA;

  auto mark = [&](int stage) -> bool {
    if (events == nullptr) return true;
    return cudaEventRecord(static_cast<cudaEvent_t>(events[stage]), stream) == cudaSuccess;
  };
  auto fail = [](cudaError_t e) { return e != cudaSuccess; };

  if (clear_flags && fail(cudaMemsetAsync(ra.flags, 0, 256, stream))) return SOLO_ERR_CUDA;

  if (!mark(SOLO_STAGE_RMSNORM) || fail(launch_keep_scan(ra, stream)) ||
      fail(launch_rmsnorm_fwd(ra, stream)))
    return SOLO_ERR_CUDA;

  GemmArgs g;
  std::memset(&g, 0, sizeof(g));
  g.M = static_cast<int32_t>(M);
  g.N = D.V;
  g.k_blocks = static_cast<int32_t>((d + kBK - 1) / kBK);
  g.k_row0 = 0;
  g.m_blocks = static_cast<int32_t>((M + 2 * kBM - 1) / (2 * kBM));
  g.n_blocks = L.n_tiles_v;
  g.group_m = kGroupLogits;
  g.num_tiles = g.m_blocks * g.n_blocks;
  g.targets = ra.tgt_c;             // compact rows: kept tokens only
  g.m_dev = ra.offsets + D.K;       // their count
  g.orig_row = ra.orig_row;
  g.stats = ra.stats;
  g.zy = ra.zy;
  g.V = D.V;
  g.flags = ra.flags;
  g.tau = tau;
  g.bias = bias;
  g.tokens_per_module = D.N;
  g.usum = ra.usum;
  g.sy = ra.sy;
  g.aux_slots = L.aux_slots;
  plan_units(g, sms, false);
  if (!mark(SOLO_STAGE_LOGITS) ||
      fail(launch_gemm(affine ? kLogitsHeads : kLogits, mX_k, mW_k, mP_st, mAux, g, sms,
                       stream)))
    return SOLO_ERR_CUDA;

  if (!mark(SOLO_STAGE_LSE) || fail(launch_lse(ra, stream, dtau != nullptr)))
    return SOLO_ERR_CUDA;
  if (!mark(SOLO_STAGE_GRAD) || fail(launch_grad(ra, stream))) return SOLO_ERR_CUDA;

  GemmArgs gx = g;
  gx.N = D.d;
  gx.k_blocks = (D.V + kBK - 1) / kBK;
  gx.n_blocks = static_cast<int32_t>((d + kBN - 1) / kBN);
  gx.group_m = kGroupDxhat;
  gx.num_tiles = gx.m_blocks * gx.n_blocks;
  // the RMSNorm backward in the epilogue (dH, and dgamma partials when wanted)
  gx.norm_fused = 1;
  gx.modules = D.K;
  for (int k = 0; k < D.K; ++k) {
    gx.hidden[k] = ra.hidden[k];
    gx.dhidden[k] = ra.dhidden[k];
  }
  gx.gamma = ra.gamma;
  gx.r = ra.r;
  gx.edz = ra.edz;
  gx.inv_nvalid = ra.inv_nvalid;
  gx.dg_part = dgamma ? ra.dgamma_part : nullptr;
  gx.dg_blocks = L.dg_chunks;
  gx.dg_row0 = static_cast<int64_t>(D.K - 1) * D.N;
  gx.row0_dev = ra.offsets + (D.K - 1);   // the final module's first kept token
  gx.row_fa = ra.row_fa;
  gx.row_fb = ra.row_fb;
  gx.W = W;
  gx.Vw = D.V;
  gx.aux_part0 = 1;     // cut tiles: every part to a slot, summed by cut_tiles_norm
  plan_units(gx, sms, true);
  // whole tiles write dH from TMEM and cut tiles write slots: the output map
  // is never used (any valid map fills its place)
  if (!mark(SOLO_STAGE_DXHAT) || fail(launch_gemm(kDxhat, mG_k, mW_mn, mAux, mAux, gx, sms, stream)))
    return SOLO_ERR_CUDA;

  if (!mark(SOLO_STAGE_NORM_BWD) || fail(launch_cut_tiles_norm(gx, aux, stream)))
    return SOLO_ERR_CUDA;

  if (!mark(SOLO_STAGE_DW)) return SOLO_ERR_CUDA;
  if (dW) {
    GemmArgs gw = g;
    gw.M = D.V;
    gw.N = D.d;
    gw.k_blocks = static_cast<int32_t>((D.N + kBK - 1) / kBK);
    gw.k_row0 = static_cast<int32_t>(static_cast<int64_t>(D.K - 1) * D.N);
    gw.m_blocks = (D.V + 2 * kBM - 1) / (2 * kBM);
    gw.n_blocks = static_cast<int32_t>((d + kBN - 1) / kBN);
    gw.group_m = kGroupDW;
    gw.num_tiles = gw.m_blocks * gw.n_blocks;
    gw.aux_part0 = 0;
    // the reduction runs over rows [offsets[K-1], offsets[K-1] + N): the final
    // module's kept tokens, then zeroed rows (masked tokens' share of [Mk, M))
    gw.m_dev = nullptr;
    gw.row0_dev = ra.offsets + (D.K - 1);
    gw.kend_dev = ra.offsets + D.K;       // the final module's kept tokens only
    gw.orig_row = nullptr;
    plan_units(gw, sms, true);
    if (fail(launch_gemm(kDW, mG_mn, mX_mn, mDW, mAux, gw, sms, stream)) ||
        fail(launch_split_fixup(gw, dW, D.d, aux, stream)))
      return SOLO_ERR_CUDA;
  }
  if (!mark(SOLO_STAGE_DGAMMA)) return SOLO_ERR_CUDA;
  if (dgamma && fail(launch_dgamma_reduce(ra, stream))) return SOLO_ERR_CUDA;
  if (!mark(SOLO_NUM_STAGES)) return SOLO_ERR_CUDA;
  return SOLO_OK;
}

// ---- exit readout (forward only) --------------------------------------------------

struct ExitLayout {
  int64_t M = 0;
  int n_tiles_v = 0;
  int part_blocks = 0;
  size_t flags = 0, r = 0, zy = 0, part_sum = 0, part_cnt = 0, inv_nvalid = 0;
  size_t stats = 0, argmax = 0, xhat = 0, total = 0;
};

ExitLayout make_exit_layout(const solo_dims_t& d) {
  ExitLayout L;
  L.M = static_cast<int64_t>(d.K) * d.N;
  L.n_tiles_v = (d.V + kBN - 1) / kBN;
  L.part_blocks = static_cast<int>((d.N + 255) / 256);
  const size_t M = static_cast<size_t>(L.M);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, kAlign);
    return at;
  };
  L.flags = take(256);
  L.r = take(M * 4);
  L.zy = take(M * 4);
  L.part_sum = take(static_cast<size_t>(d.K) * L.part_blocks * 8);
  L.part_cnt = take(static_cast<size_t>(d.K) * L.part_blocks * 4);
  L.inv_nvalid = take(SOLO_MAX_MODULES * 4);
  L.stats = take(static_cast<size_t>(L.n_tiles_v) * M * 8);
  L.argmax = take(static_cast<size_t>(L.n_tiles_v) * M * 4);
  L.xhat = take(M * d.d * 2);
  L.total = off;
  return L;
}

solo_status_t run_exit(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                       const solo_bf16_t* gamma, const solo_bf16_t* W, const int32_t* targets,
                       const uint8_t* mask, float* loss_tok, float* loss_mean, int32_t* top1,
                       float* top1_logprob, void* workspace, size_t workspace_bytes,
                       cudaStream_t stream, void* const* events, int32_t n_events) {
  solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  const solo_dims_t& D = *dims;
  if (hidden == nullptr || gamma == nullptr || W == nullptr || workspace == nullptr)
    return SOLO_ERR_INVALID_ARG;
  if (targets == nullptr && (loss_tok != nullptr || loss_mean != nullptr))
    return SOLO_ERR_INVALID_ARG;     // losses need targets
  if (events != nullptr && n_events != SOLO_EXIT_NUM_STAGES + 1) return SOLO_ERR_INVALID_ARG;
  for (int k = 0; k < D.K; ++k) {
    if (hidden[k] == nullptr) return SOLO_ERR_INVALID_ARG;
    if (!aligned16(hidden[k])) return SOLO_ERR_MISALIGNED;
  }
  auto a4 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; };
  if (!aligned16(gamma) || !aligned16(W) || !aligned16(workspace) || !a4(targets) ||
      !a4(loss_tok) || !a4(loss_mean) || !a4(top1) || !a4(top1_logprob))
    return SOLO_ERR_MISALIGNED;
  const ExitLayout L = make_exit_layout(D);
  if (workspace_bytes < L.total) return SOLO_ERR_WORKSPACE_TOO_SMALL;
  {
    const size_t K = static_cast<size_t>(D.K), N = static_cast<size_t>(D.N);
    Ranges rg;
    for (int k = 0; k < D.K; ++k) rg.add(hidden[k], N * D.d * 2, false);
    rg.add(gamma, static_cast<size_t>(D.d) * 2, false);
    rg.add(W, static_cast<size_t>(D.V) * D.d * 2, false);
    rg.add(targets, K * N * 4, false);
    rg.add(mask, K * N, false);
    rg.add(loss_tok, K * N * 4, true);
    rg.add(loss_mean, K * 4, true);
    rg.add(top1, K * N * 4, true);
    rg.add(top1_logprob, K * N * 4, true);
    rg.add(workspace, L.total, true);
    if (rg.any_output_overlap()) return SOLO_ERR_INVALID_ARG;
  }
  int sms = 0;
  st = device_setup(&sms);
  if (st != SOLO_OK) return st;

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  RowArgs ra;
  std::memset(&ra, 0, sizeof(ra));
  for (int k = 0; k < D.K; ++k) ra.hidden[k] = hidden[k];
  ra.N = D.N;
  ra.K = D.K;
  ra.d = D.d;
  ra.V = D.V;
  ra.n_tiles_v = L.n_tiles_v;
  ra.ignore_index = D.ignore_index;
  ra.eps = D.eps;
  ra.gamma = gamma;
  ra.targets = targets;
  ra.mask = mask;
  ra.r = reinterpret_cast<float*>(ws + L.r);
  ra.xhat = reinterpret_cast<uint16_t*>(ws + L.xhat);
  ra.zy = reinterpret_cast<float*>(ws + L.zy);
  ra.stats = reinterpret_cast<float2*>(ws + L.stats);
  ra.part_sum = reinterpret_cast<double*>(ws + L.part_sum);
  ra.part_cnt = reinterpret_cast<int32_t*>(ws + L.part_cnt);
  ra.part_blocks = L.part_blocks;
  ra.inv_nvalid = reinterpret_cast<float*>(ws + L.inv_nvalid);
  ra.loss_tok = loss_tok;
  ra.loss_mean = loss_mean;
  ra.flags = reinterpret_cast<uint32_t*>(ws + L.flags);
  ra.argmax = reinterpret_cast<int32_t*>(ws + L.argmax);
  ra.top1 = top1;
  ra.top1_logprob = top1_logprob;

  const uint64_t M = static_cast<uint64_t>(L.M);
  const uint64_t d = static_cast<uint64_t>(D.d);
  const uint64_t V = static_cast<uint64_t>(D.V);
  CUtensorMap mX_k, mW_k;
  if (!make_map(&mX_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ra.xhat, d, M, d * 2, 64, kBM) ||
      !make_map(&mW_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, W, d, V, d * 2, 64, kBN / 2))
    return SOLO_ERR_CUDA;
  auto mark = [&](int stage) -> bool {
    if (events == nullptr) return true;
    return cudaEventRecord(static_cast<cudaEvent_t>(events[stage]), stream) == cudaSuccess;
  };
  if (cudaMemsetAsync(ra.flags, 0, 256, stream) != cudaSuccess) return SOLO_ERR_CUDA;
  if (!mark(0) || launch_rmsnorm_fwd(ra, stream) != cudaSuccess) return SOLO_ERR_CUDA;
  GemmArgs g;
  std::memset(&g, 0, sizeof(g));
  g.M = static_cast<int32_t>(M);
  g.N = D.V;
  g.k_blocks = static_cast<int32_t>((d + kBK - 1) / kBK);
  g.m_blocks = static_cast<int32_t>((M + 2 * kBM - 1) / (2 * kBM));
  g.n_blocks = L.n_tiles_v;
  g.group_m = kGroupLogits;
  g.num_tiles = g.m_blocks * g.n_blocks;
  plan_units(g, sms, false);
  g.targets = targets;
  g.stats = ra.stats;
  g.zy = ra.zy;
  g.V = D.V;
  g.flags = ra.flags;
  g.argmax = ra.argmax;
  // the store map is unused by this epilogue; any valid map fills the slot
  if (!mark(1) || launch_gemm(kExit, mX_k, mW_k, mX_k, mX_k, g, sms, stream) != cudaSuccess)
    return SOLO_ERR_CUDA;
  if (!mark(2) || launch_exit_lse(ra, stream) != cudaSuccess) return SOLO_ERR_CUDA;
  if (!mark(3)) return SOLO_ERR_CUDA;
  return SOLO_OK;
}

// ---- on-chip backward of the auxiliary modules ----------------------------------

struct OnchipLayout {
  size_t final_total = 0;     // the final module's stored-path layout, at offset 0
  size_t xhat = 0, r = 0, row_loss = 0, n_valid = 0, inv_nvalid = 0, total = 0;
};

OnchipLayout make_onchip_layout(const solo_dims_t& d) {
  OnchipLayout L;
  solo_dims_t one = d;
  one.K = 1;
  L.final_total = make_layout(one).total;
  const size_t Maux = static_cast<size_t>(d.K - 1) * static_cast<size_t>(d.N);
  size_t off = align_up(L.final_total, kAlign);
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, kAlign);
    return at;
  };
  L.xhat = take(Maux * d.d * 2);
  L.r = take(Maux * 4);
  L.row_loss = take(Maux * 4);
  L.n_valid = take(SOLO_MAX_MODULES * 4);
  L.inv_nvalid = take(SOLO_MAX_MODULES * 4);
  L.total = off;
  return L;
}

solo_status_t check_onchip_dims(const solo_dims_t* dims) {
  const solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  if (dims->d > kFlashMaxD) return SOLO_ERR_UNSUPPORTED_SHAPE;
  return SOLO_OK;
}

solo_status_t run_onchip(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                         const solo_bf16_t* gamma, const solo_bf16_t* W, const int32_t* targets,
                         const uint8_t* mask, float* loss_tok, float* loss_mean,
                         solo_bf16_t* const* dhidden, float* dW, float* dgamma, void* workspace,
                         size_t workspace_bytes, cudaStream_t stream, void* const* events,
                         int32_t n_events) {
  solo_status_t st = check_onchip_dims(dims);
  if (st != SOLO_OK) return st;
  const solo_dims_t& D = *dims;
  if (hidden == nullptr || dhidden == nullptr || gamma == nullptr || W == nullptr ||
      targets == nullptr || loss_mean == nullptr || workspace == nullptr)
    return SOLO_ERR_INVALID_ARG;
  if (events != nullptr && n_events != SOLO_ONCHIP_NUM_STAGES + 1) return SOLO_ERR_INVALID_ARG;
  for (int k = 0; k < D.K; ++k) {
    if (hidden[k] == nullptr || dhidden[k] == nullptr) return SOLO_ERR_INVALID_ARG;
    if (!aligned16(hidden[k]) || !aligned16(dhidden[k])) return SOLO_ERR_MISALIGNED;
  }
  if (!aligned16(gamma) || !aligned16(W) || !aligned16(workspace) ||
      (reinterpret_cast<uintptr_t>(targets) & 3u) || (dW && !aligned16(dW)) ||
      (dgamma && (reinterpret_cast<uintptr_t>(dgamma) & 3u)) ||
      (loss_tok && (reinterpret_cast<uintptr_t>(loss_tok) & 3u)) ||
      (reinterpret_cast<uintptr_t>(loss_mean) & 3u))
    return SOLO_ERR_MISALIGNED;
  const OnchipLayout L = make_onchip_layout(D);
  if (workspace_bytes < L.total) return SOLO_ERR_WORKSPACE_TOO_SMALL;
  {
    const size_t K = static_cast<size_t>(D.K), N = static_cast<size_t>(D.N);
    const size_t dd = static_cast<size_t>(D.d), VV = static_cast<size_t>(D.V);
    Ranges rg;
    for (int k = 0; k < D.K; ++k) {
      rg.add(hidden[k], N * dd * 2, false);
      rg.add(dhidden[k], N * dd * 2, true);
    }
    rg.add(gamma, dd * 2, false);
    rg.add(W, VV * dd * 2, false);
    rg.add(targets, K * N * 4, false);
    rg.add(mask, K * N, false);
    rg.add(loss_tok, K * N * 4, true);
    rg.add(loss_mean, K * 4, true);
    rg.add(dW, VV * dd * 4, true);
    rg.add(dgamma, dd * 4, true);
    rg.add(workspace, L.total, true);
    if (rg.any_output_overlap()) return SOLO_ERR_INVALID_ARG;
  }
  int sms = 0, dev = 0;
  st = device_setup(&sms, &dev);
  if (st != SOLO_OK) return st;
  auto mark = [&](int stage) -> bool {
    if (events == nullptr) return true;
    return cudaEventRecord(static_cast<cudaEvent_t>(events[stage]), stream) == cudaSuccess;
  };

  // 1. the final module on the stored path (it needs G for dW); clears the flags
  const int64_t kf = D.K - 1;
  solo_dims_t one = D;
  one.K = 1;
  if (!mark(SOLO_ONCHIP_STAGE_FINAL)) return SOLO_ERR_CUDA;
  st = run(&one, hidden + kf, gamma, W, targets + kf * D.N, mask ? mask + kf * D.N : nullptr,
           nullptr, loss_tok ? loss_tok + kf * D.N : nullptr, loss_mean + kf, dhidden + kf, dW,
           dgamma, workspace, L.final_total, stream, nullptr, 0, /*clear_flags=*/true);
  if (st != SOLO_OK) return st;

  // 2. the auxiliary modules in one on-chip pass
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const int aux = D.K - 1;
  FlashArgs fa;
  std::memset(&fa, 0, sizeof(fa));
  fa.M = static_cast<int32_t>(static_cast<int64_t>(aux) * D.N);
  fa.d = D.d;
  fa.V = D.V;
  fa.ds = flash_slice_width(D.d);
  fa.n_tiles = (D.V + 63) / 64;
  fa.row_blocks = static_cast<int32_t>((static_cast<int64_t>(fa.M) + 127) / 128);
  fa.N = D.N;
  fa.modules = aux;
  fa.ignore_index = D.ignore_index;
  fa.targets = targets;
  fa.mask = mask;
  fa.xhat = reinterpret_cast<const uint16_t*>(ws + L.xhat);
  fa.r = reinterpret_cast<const float*>(ws + L.r);
  float* inv_nvalid = reinterpret_cast<float*>(ws + L.inv_nvalid);
  fa.inv_nvalid = inv_nvalid;
  fa.W = W;
  fa.gamma = gamma;
  for (int k = 0; k < aux; ++k) {
    fa.hidden[k] = hidden[k];
    fa.dhidden[k] = dhidden[k];
  }
  fa.loss_tok = loss_tok;
  fa.row_loss = reinterpret_cast<float*>(ws + L.row_loss);
  fa.n_valid = reinterpret_cast<int32_t*>(ws + L.n_valid);
  fa.loss_mean = loss_mean;
  fa.flags = reinterpret_cast<uint32_t*>(ws);     // the final module's flag word
  if (!mark(SOLO_ONCHIP_STAGE_AUX_PREP)) return SOLO_ERR_CUDA;
  CUtensorMap mW;
  if (aux > 0) {
    RowArgs ra;
    std::memset(&ra, 0, sizeof(ra));
    for (int k = 0; k < aux; ++k) ra.hidden[k] = hidden[k];
    ra.N = D.N;
    ra.K = aux;
    ra.d = D.d;
    ra.V = D.V;
    ra.eps = D.eps;
    ra.gamma = gamma;
    ra.xhat = reinterpret_cast<uint16_t*>(ws + L.xhat);
    ra.r = reinterpret_cast<float*>(ws + L.r);
    ra.flags = fa.flags;
    if (launch_rmsnorm_fwd(ra, stream) != cudaSuccess ||
        launch_flash_count(fa, inv_nvalid, stream) != cudaSuccess)
      return SOLO_ERR_CUDA;
    if (!make_map(&mW, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, W, static_cast<uint64_t>(D.d),
                  static_cast<uint64_t>(D.V), static_cast<uint64_t>(D.d) * 2, 64, 64))
      return SOLO_ERR_CUDA;
  }
  if (!mark(SOLO_ONCHIP_STAGE_AUX)) return SOLO_ERR_CUDA;
  if (aux > 0 && launch_flash(mW, fa, dev, sms, stream) != cudaSuccess) return SOLO_ERR_CUDA;
  if (!mark(SOLO_ONCHIP_STAGE_AUX_MEANS)) return SOLO_ERR_CUDA;
  if (aux > 0 && launch_flash_means(fa, stream) != cudaSuccess) return SOLO_ERR_CUDA;
  if (!mark(SOLO_ONCHIP_NUM_STAGES)) return SOLO_ERR_CUDA;
  return SOLO_OK;
}

}  // namespace

extern "C" {

solo_status_t solo_readout_onchip_workspace_bytes(const solo_dims_t* dims, size_t* bytes) {
  if (bytes == nullptr) return SOLO_ERR_INVALID_ARG;
  const solo_status_t st = check_onchip_dims(dims);
  if (st != SOLO_OK) return st;
  *bytes = make_onchip_layout(*dims).total;
  return SOLO_OK;
}

solo_status_t solo_readout_fwd_bwd_onchip(const solo_dims_t* dims,
                                          const solo_bf16_t* const* hidden,
                                          const solo_bf16_t* gamma, const solo_bf16_t* W,
                                          const int32_t* targets, const uint8_t* mask,
                                          float* loss_tok, float* loss_mean,
                                          solo_bf16_t* const* dhidden, float* dW, float* dgamma,
                                          void* workspace, size_t workspace_bytes,
                                          solo_stream_t stream, void* const* events,
                                          int32_t n_events) {
  return run_onchip(dims, hidden, gamma, W, targets, mask, loss_tok, loss_mean, dhidden, dW,
                    dgamma, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream),
                    events, events ? n_events : 0);
}

solo_status_t solo_readout_workspace_bytes(const solo_dims_t* dims, size_t* bytes) {
  if (bytes == nullptr) return SOLO_ERR_INVALID_ARG;
  const solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  *bytes = make_layout(*dims).total;
  return SOLO_OK;
}

solo_status_t solo_readout_fwd_bwd(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                                   const solo_bf16_t* gamma, const solo_bf16_t* W,
                                   const int32_t* targets, const uint8_t* mask, float* loss_tok,
                                   float* loss_mean, solo_bf16_t* const* dhidden, float* dW,
                                   float* dgamma, void* workspace, size_t workspace_bytes,
                                   solo_stream_t stream) {
  return run(dims, hidden, gamma, W, targets, mask, nullptr, loss_tok, loss_mean, dhidden, dW,
             dgamma, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), nullptr,
             0);
}

solo_status_t solo_readout_fwd_bwd_heads(const solo_dims_t* dims,
                                         const solo_bf16_t* const* hidden,
                                         const solo_bf16_t* gamma, const solo_bf16_t* W,
                                         const int32_t* targets, const uint8_t* mask,
                                         const solo_heads_t* heads, float* loss_tok,
                                         float* loss_mean, solo_bf16_t* const* dhidden,
                                         float* dW, float* dgamma, void* workspace,
                                         size_t workspace_bytes, solo_stream_t stream,
                                         void* const* events, int32_t n_events) {
  return run(dims, hidden, gamma, W, targets, mask, heads, loss_tok, loss_mean, dhidden, dW,
             dgamma, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), events,
             events ? n_events : 0);
}

solo_status_t solo_readout_fwd_bwd_events(const solo_dims_t* dims,
                                          const solo_bf16_t* const* hidden,
                                          const solo_bf16_t* gamma, const solo_bf16_t* W,
                                          const int32_t* targets, const uint8_t* mask,
                                          float* loss_tok, float* loss_mean,
                                          solo_bf16_t* const* dhidden, float* dW, float* dgamma,
                                          void* workspace, size_t workspace_bytes,
                                          solo_stream_t stream, void* const* events,
                                          int32_t n_events) {
  if (events == nullptr) return SOLO_ERR_INVALID_ARG;
  return run(dims, hidden, gamma, W, targets, mask, nullptr, loss_tok, loss_mean, dhidden, dW,
             dgamma, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), events,
             n_events);
}

solo_status_t solo_readout_exit_workspace_bytes(const solo_dims_t* dims, size_t* bytes) {
  if (bytes == nullptr) return SOLO_ERR_INVALID_ARG;
  const solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  *bytes = make_exit_layout(*dims).total;
  return SOLO_OK;
}

solo_status_t solo_readout_exit_forward(const solo_dims_t* dims,
                                        const solo_bf16_t* const* hidden,
                                        const solo_bf16_t* gamma, const solo_bf16_t* W,
                                        const int32_t* targets, const uint8_t* mask,
                                        float* loss_tok, float* loss_mean, int32_t* top1,
                                        float* top1_logprob, void* workspace,
                                        size_t workspace_bytes, solo_stream_t stream) {
  return run_exit(dims, hidden, gamma, W, targets, mask, loss_tok, loss_mean, top1,
                  top1_logprob, workspace, workspace_bytes,
                  reinterpret_cast<cudaStream_t>(stream), nullptr, 0);
}

solo_status_t solo_readout_exit_forward_events(
    const solo_dims_t* dims, const solo_bf16_t* const* hidden, const solo_bf16_t* gamma,
    const solo_bf16_t* W, const int32_t* targets, const uint8_t* mask, float* loss_tok,
    float* loss_mean, int32_t* top1, float* top1_logprob, void* workspace,
    size_t workspace_bytes, solo_stream_t stream, void* const* events, int32_t n_events) {
  if (events == nullptr) return SOLO_ERR_INVALID_ARG;
  return run_exit(dims, hidden, gamma, W, targets, mask, loss_tok, loss_mean, top1,
                  top1_logprob, workspace, workspace_bytes,
                  reinterpret_cast<cudaStream_t>(stream), events, n_events);
}

solo_status_t solo_readout_private_workspace_bytes(const solo_dims_t* dims, size_t* bytes) {
  if (bytes == nullptr) return SOLO_ERR_INVALID_ARG;
  solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  solo_dims_t one = *dims;
  one.K = 1;
  *bytes = make_layout(one).total;
  return SOLO_OK;
}

solo_status_t solo_readout_fwd_bwd_private(
    const solo_dims_t* dims, const solo_bf16_t* const* hidden, const solo_bf16_t* const* gamma,
    const solo_bf16_t* const* W, const int32_t* targets, const uint8_t* mask,
    const solo_heads_t* heads, float* loss_tok, float* loss_mean, solo_bf16_t* const* dhidden,
    float* const* dW, float* const* dgamma, void* workspace, size_t workspace_bytes,
    solo_stream_t stream) {
  solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  const solo_dims_t D = *dims;
  if (hidden == nullptr || gamma == nullptr || W == nullptr || dhidden == nullptr ||
      targets == nullptr || loss_mean == nullptr)
    return SOLO_ERR_INVALID_ARG;
  for (int k = 0; k < D.K; ++k)
    if (gamma[k] == nullptr || W[k] == nullptr || hidden[k] == nullptr || dhidden[k] == nullptr)
      return SOLO_ERR_INVALID_ARG;
  solo_dims_t one = D;
  one.K = 1;
  if (workspace_bytes < make_layout(one).total) return SOLO_ERR_WORKSPACE_TOO_SMALL;
  // Every module is its own single-module problem: its head's readout W_k and
  // final-norm gain gamma_k, with dW_k and dgamma_k.  The modules run one after
  // another on `stream` and share the workspace; device flags accumulate.
  const int64_t N = D.N;
  for (int k = 0; k < D.K; ++k) {
    solo_heads_t hk{};
    const solo_heads_t* hp = nullptr;
    if (heads) {
      hk.tau = heads->tau ? heads->tau + k : nullptr;
      hk.bias = heads->bias ? heads->bias + static_cast<int64_t>(k) * D.V : nullptr;
      hk.dtau = heads->dtau ? heads->dtau + k : nullptr;
      hk.dbias = heads->dbias ? heads->dbias + static_cast<int64_t>(k) * D.V : nullptr;
      hp = &hk;
    }
    st = run(&one, hidden + k, gamma[k], W[k], targets + k * N, mask ? mask + k * N : nullptr,
             hp, loss_tok ? loss_tok + k * N : nullptr, loss_mean + k, dhidden + k,
             dW ? dW[k] : nullptr, dgamma ? dgamma[k] : nullptr, workspace, workspace_bytes,
             reinterpret_cast<cudaStream_t>(stream), nullptr, 0, /*clear_flags=*/k == 0);
    if (st != SOLO_OK) return st;
  }
  return SOLO_OK;
}

solo_status_t solo_readout_rmsnorm(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                                   const solo_bf16_t* gamma, solo_bf16_t* xhat, float* r,
                                   solo_stream_t stream) {
  solo_status_t st = check_dims(dims);
  if (st != SOLO_OK) return st;
  const solo_dims_t& D = *dims;
  if (hidden == nullptr || gamma == nullptr || xhat == nullptr) return SOLO_ERR_INVALID_ARG;
  for (int k = 0; k < D.K; ++k) {
    if (hidden[k] == nullptr) return SOLO_ERR_INVALID_ARG;
    if (!aligned16(hidden[k])) return SOLO_ERR_MISALIGNED;
  }
  if (!aligned16(gamma) || !aligned16(xhat) || (reinterpret_cast<uintptr_t>(r) & 3u))
    return SOLO_ERR_MISALIGNED;
  {
    const size_t M = static_cast<size_t>(D.K) * D.N;
    Ranges rg;
    for (int k = 0; k < D.K; ++k) rg.add(hidden[k], static_cast<size_t>(D.N) * D.d * 2, false);
    rg.add(gamma, static_cast<size_t>(D.d) * 2, false);
    rg.add(xhat, M * D.d * 2, true);
    rg.add(r, M * 4, true);
    if (rg.any_output_overlap()) return SOLO_ERR_INVALID_ARG;
  }
  int sms = 0;
  st = device_setup(&sms);
  if (st != SOLO_OK) return st;
  RowArgs ra;
  std::memset(&ra, 0, sizeof(ra));
  for (int k = 0; k < D.K; ++k) ra.hidden[k] = hidden[k];
  ra.N = D.N;
  ra.K = D.K;
  ra.d = D.d;
  ra.V = D.V;
  ra.eps = D.eps;
  ra.gamma = gamma;
  ra.xhat = xhat;
  ra.r = r;
  return launch_rmsnorm_fwd(ra, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? SOLO_OK
             : SOLO_ERR_CUDA;
}

solo_status_t solo_readout_get_flags(const void* workspace, solo_stream_t stream,
                                     uint32_t* flags) {
  if (workspace == nullptr || flags == nullptr) return SOLO_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint32_t v = 0;
  if (cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return SOLO_ERR_CUDA;
  *flags = v;
  return SOLO_OK;
}

const char* solo_readout_strerror(solo_status_t status) {
  switch (status) {
    case SOLO_OK: return "success";
    case SOLO_ERR_INVALID_ARG: return "invalid argument (NULL pointer or dims out of range)";
    case SOLO_ERR_UNSUPPORTED_SHAPE:
      return "unsupported shape (d must be a multiple of 8; V at most 2^23; K*N and the "
             "tile counts within 32-bit coordinates)";
    case SOLO_ERR_WORKSPACE_TOO_SMALL: return "workspace smaller than solo_readout_workspace_bytes";
    case SOLO_ERR_CUDA: return "a CUDA runtime call failed";
    case SOLO_ERR_NOT_SM103: return "current device is not compute capability 10.3 (sm_103a)";
    case SOLO_ERR_MISALIGNED: return "a tensor pointer is not suitably aligned (16 bytes)";
    case SOLO_ERR_EXCEEDS_STATIC_SCRATCH:
      return "problem needs more scratch than the 64 MiB built-in array of "
             "solo_readout_fwd_bwd_static; use solo_readout_fwd_bwd with a workspace";
    default: return "unknown status";
  }
}

int32_t solo_readout_version(void) { return 100; }

uint64_t solo_readout_kernel_launches(void) { return solo::launch_count(); }

int32_t solo_readout_build_flags(void) { return SOLO_DEBUG ? SOLO_BUILD_CHECKED : 0; }

}  // extern "C"

// ---- allocation-free variant -----------------------------------------------------
// For callers that cannot allocate device memory.  The scratch that
// solo_readout_fwd_bwd takes from the caller's workspace comes instead from a
// fixed array compiled into this file's device code.  In host code the name
// g_static_scratch is only a host-side stand-in for the symbol, so its device
// address is looked up per device with cudaGetSymbolAddress (on the first call
// on that device) and that address is what the kernels receive.

namespace {

static __device__ __align__(256) unsigned char g_static_scratch[SOLO_STATIC_SCRATCH_BYTES];

std::mutex g_static_mu;
void* g_static_ptr[64] = {};

// Device address of the scratch array on the current device, looked up once.
solo_status_t static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SOLO_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (g_static_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
      return SOLO_ERR_CUDA;
    g_static_ptr[dev] = p;
  }
  *out = g_static_ptr[dev];
  return SOLO_OK;
}

}  // namespace

extern "C" solo_status_t solo_readout_fwd_bwd_static(
    const solo_dims_t* dims, const solo_bf16_t* const* hidden, const solo_bf16_t* gamma,
    const solo_bf16_t* W, const int32_t* targets, const uint8_t* mask, float* loss_tok,
    float* loss_mean, solo_bf16_t* const* dhidden, float* dW, float* dgamma,
    uint32_t* device_flags, solo_stream_t stream) {
  size_t need = 0;
  solo_status_t st = solo_readout_workspace_bytes(dims, &need);
  if (st != SOLO_OK) return st;
  if (need > SOLO_STATIC_SCRATCH_BYTES) return SOLO_ERR_EXCEEDS_STATIC_SCRATCH;
  if (device_flags && (reinterpret_cast<uintptr_t>(device_flags) & 3u)) return SOLO_ERR_MISALIGNED;
  void* scratch = nullptr;
  st = static_scratch_address(&scratch);
  if (st != SOLO_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // The launch sequence clears the flag word itself; every other scratch
  // buffer is written before it is read, so stale contents never leak.
  st = run(dims, hidden, gamma, W, targets, mask, nullptr, loss_tok, loss_mean, dhidden, dW,
           dgamma, scratch, SOLO_STATIC_SCRATCH_BYTES, s, nullptr, 0);
  if (st != SOLO_OK) return st;
  if (device_flags &&
      cudaMemcpyAsync(device_flags, scratch, sizeof(uint32_t), cudaMemcpyDeviceToDevice, s) !=
          cudaSuccess)
    return SOLO_ERR_CUDA;
  return SOLO_OK;
}
