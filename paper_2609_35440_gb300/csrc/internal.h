// Declarations shared by the translation units of libsolo_readout.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#ifndef SOLO_DEBUG
#define SOLO_DEBUG 0
#endif

namespace solo {

// Checked builds (SOLO_DEBUG = 1) test computed global indices against the
// extent of their buffer; a failed test sets SOLO_FLAG_BOUNDS (4) in the flag
// word and the caller skips the access.  Release builds compile the tests away.
__device__ __forceinline__ bool in_bounds(bool ok, uint32_t* flags) {
#if SOLO_DEBUG
  if (!ok) atomicOr(flags, 4u);
  return ok;
#else
  (void)ok;
  (void)flags;
  return true;
#endif
}

// Every kernel launch of the library goes through launched(): it returns the
// launch's error and counts the successful ones for
// solo_readout_kernel_launches.
void note_launch();
uint64_t launch_count();
inline cudaError_t launched() {
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) note_launch();
  return e;
}

// Tensor-core tile: a CTA pair computes 256 rows x 256 columns (each CTA owns
// 128 rows), reduction in blocks of kBK through a shared-memory ring.
constexpr int kBM = 128;
constexpr int kBN = 256;
#ifndef SOLO_GEMM_BK
#define SOLO_GEMM_BK 128
#endif
constexpr int kBK = SOLO_GEMM_BK;          // 64 or 128 bf16 elements per reduction block
static_assert(kBK == 64 || kBK == 128, "reduction block");
constexpr int kStages = 6 * 64 / kBK;      // 192 KB of operand ring per CTA
constexpr int kKAtoms = kBK / 64;          // 128-byte swizzle atoms along K per row
constexpr int kGemmThreads = 192;   // warp 0: TMA, warp 1: MMA, warps 2-5: epilogue

constexpr int kMaxModules = 16;

// The products of the GEMM kernel.
enum GemmMode : int {
  kLogits = 0,  // Z = Xhat W^T (A: Xhat K-major, B: W K-major); epilogue: per-tile
                //   max / sum of exp, target logit, bf16 exp(z - tile max) stored
  kDxhat = 1,   // dXhat = G W (A: G K-major, B: W MN-major); epilogue: the RMSNorm
                //   backward into bf16 dH (norm_fused), or fp32 dXhat
  kDW = 2,      // dW = G^T Xhat over the final module (A: G MN-major,
                //   B: Xhat MN-major); epilogue: fp32 store
  kExit = 3,    // Z = Xhat W^T for decoding only; epilogue: per-tile max, sum of
                //   exp, first argmax, target logit; nothing else is stored
  kLogitsHeads = 4  // as kLogits with each head's temperature and bias applied,
                    //   z = tau_k s + b_k (s = Xhat W^T), and per tile the sum of
                    //   exp(z - m) s for the temperature's gradient
};

struct GemmArgs {
  int32_t M;          // rows of the product
  int32_t N;          // columns of the product
  int32_t k_blocks;   // reduction length / kBK, rounded up
  int32_t k_row0;     // first reduction row in A/B coordinates (kDW: first token of the module)
  int32_t m_blocks;   // 256-row blocks (one per CTA pair)
  int32_t n_blocks;   // 256-column blocks
  int32_t group_m;    // tile raster: group_m row blocks sweep all column blocks together
  int32_t num_tiles;
  // Work units: tiles [0, full_tiles) whole, then each remaining tile cut
  // into `split` contiguous reduction ranges (fills the last partial wave of
  // CTA pairs).  Part 0 of a cut tile is stored to the output, parts 1.. to
  // the auxiliary buffer (slot (tile - full_tiles) * (split - 1) + part - 1,
  // 256 x 256 fp32 each) and added by launch_split_fixup in a fixed order
  // (with aux_part0, every part goes to the auxiliary buffer).
  int32_t full_tiles;
  int32_t split;
  int32_t num_units;
  int32_t aux_slots;       // slots in the auxiliary buffer
  int32_t aux_part0;       // 1: part 0 of a cut tile goes to the auxiliary buffer as
                           //   well (slot (tile - full_tiles) * split + part), and the
                           //   output is never written for cut tiles (kDxhat with the
                           //   fused RMSNorm backward: cut_tiles_norm sums the parts)
  // kLogits epilogue
  const int32_t* targets;  // [M] token targets (flattened [K, N])
  float2* stats;           // [n_blocks, M]: (max, sum exp(z - max)) per tile; kLogits /
                           //   kLogitsHeads leave the target's own term out of the sum
  float* zy;               // [M]: logit of the target
  int32_t V;
  uint32_t* flags;         // device flag word
  int32_t* argmax;         // kExit: [n_blocks, M] first column of the tile maximum
  // kLogitsHeads
  const float* tau;        // [K] or null (1)
  const float* bias;       // [K, V] or null (0)
  int64_t tokens_per_module;
  float* usum;             // [n_blocks, M]: sum over the tile of exp(z - m) * s (the
                           //   target's term left out, like the sum in stats)
  float* sy;               // [M]: s at the target (before temperature and bias)
  // kDxhat with the RMSNorm backward fused into the epilogue (norm_fused = 1):
  // whole tiles write dH = r gamma dxhat - (r^3 / d) h S in bf16 and the final
  // module's dgamma partial sums; cut tiles store their fp32 parts (aux_part0).
  int32_t norm_fused;
  int32_t modules;                       // K
  const uint16_t* hidden[kMaxModules];   // [N, d] bf16 per module
  uint16_t* dhidden[kMaxModules];        // [N, d] bf16 per module
  const uint16_t* gamma;                 // [d]
  const float* r;                        // [M]
  const float* edz;                      // [M]: E_p[s] - s_y of a kept token, else 0
  const float* inv_nvalid;               // [K]
  float* dg_part;          // [dg_blocks, d] or null: per 32-row block of the final module
  int32_t dg_blocks;
  int64_t dg_row0;         // first row of the final module
  // Compacted rows (masked tokens skipped): the row count, the final module's
  // first row and the token of each row live in device memory.  With m_dev the
  // kernel plans its tiles and cut tiles itself from *m_dev <= M (the host's
  // full_tiles / split / num_units describe the upper bound M).
  const int32_t* m_dev;     // rows of the product, or null (M)
  const int32_t* row0_dev;  // kDW: first reduction row / kDxhat: first row of the final
                            //   module (dgamma blocks), or null (k_row0 / dg_row0)
  const int32_t* orig_row;  // [M]: token (k * N + n) of a row, or null (the row itself)
  const int32_t* kend_dev;  // kDW: end of the reduction rows (the kept tokens' count):
                            //   the device plan reduces over [*row0_dev, *kend_dev)
                            //   rounded up to whole blocks, or null (k_blocks)
  int32_t sms;              // multiprocessors, for the device-side plan
  int32_t split_ok;         // the plan may cut the last partial wave
  // kDxhat: rows whose gradient the epilogue forms from the stored exponentials
  // (exp(z) against the reference 0): dxhat = tau/Nvalid (fa acc - fb W_y).
  // fa < 0 marks a row the gradient pass has turned into G (fa = 1, fb = 0).
  const float* row_fa;      // [M] e^{-lse}, or -1; null: every row is G
  const float* row_fb;      // [M] 1 - p_y
  const uint16_t* W;        // [V, d] for W_y
  int32_t Vw;               // V
};

size_t gemm_smem_bytes();
cudaError_t gemm_prepare(int device);  // sets the dynamic shared memory limit once per device

constexpr int kMaxSplit = 8;        // reduction ranges per cut tile
constexpr int kMaxAuxSlots = 127;   // 256 x 256 fp32 partial tiles (32 MB)
// Sets full_tiles / split / num_units: whole tiles fill complete waves of
// min(sms / 2, kMaxAuxSlots + 1) pairs; the remainder is cut so the last wave
// has as many units as pairs (each part keeps >= 1 reduction block) and its
// parts fit in g.aux_slots (g.aux_part0: every part takes a slot; otherwise
// part 0 goes to the output).  allow_split = false keeps every tile whole.
void plan_units(GemmArgs& g, int sms, bool allow_split);
// Slots a product needs at most: `tiles` tiles of `k_blocks` reduction
// blocks, with (part0 = true) or without part 0 in the auxiliary buffer.
inline int split_aux_slots(int64_t tiles, int64_t k_blocks, bool part0) {
  const int64_t parts = k_blocks < kMaxSplit ? k_blocks : kMaxSplit;
  const int64_t s = tiles * (part0 ? parts : parts - 1);
  return static_cast<int>(s < kMaxAuxSlots ? s : kMaxAuxSlots);
}
// Launches min(units, sms / 2) CTA pairs.  x: tensor map of the auxiliary
// buffer (fp32 [slots * 256, 256], 32 x 32 boxes) for the cut tiles' parts.
cudaError_t launch_gemm(GemmMode mode, const CUtensorMap& a, const CUtensorMap& b,
                        const CUtensorMap& d, const CUtensorMap& x, const GemmArgs& args,
                        int sms, cudaStream_t stream);
// out (fp32, row stride ld) += the auxiliary parts of every cut tile.
cudaError_t launch_split_fixup(const GemmArgs& g, float* out, int64_t ld, const float* aux,
                               cudaStream_t stream);
// kDxhat with norm_fused (and aux_part0): the RMSNorm backward (dH, dgamma
// partials) of the cut tiles, from the sum of their parts in the auxiliary
// buffer, added in part order.
cudaError_t launch_cut_tiles_norm(const GemmArgs& g, const float* aux, cudaStream_t stream);

// ---- single-pass on-chip backward of the auxiliary modules ------------------------
// dxhat_i = (sum over v != y of exp(z_v - m) W_v) / S - (S' / S) W_y (Eq. 3 with the
// softmax written out; S = sum over all v of exp(z_v - m), S' the same without the
// target), accumulated over the vocabulary with the logits kept on chip.  A
// cluster of C CTAs shares a block of 128 rows; CTA c owns the d-columns
// [c * ds, c * ds + ds) of dxhat.

struct FlashArgs {
  int32_t M;             // auxiliary rows (K - 1 modules of N tokens, module-major)
  int32_t d;
  int32_t V;
  int32_t ds;            // d-columns per CTA (multiple of 64, <= 256)
  int32_t n_tiles;       // 64-column vocabulary tiles
  int32_t row_blocks;    // 128-row blocks
  int64_t N;             // tokens per module
  int32_t modules;       // auxiliary modules (K - 1)
  int32_t ignore_index;
  const int32_t* targets;   // [M]
  const uint8_t* mask;      // [M] or null
  const uint16_t* xhat;     // [M, d] bf16
  const float* r;           // [M]
  const float* inv_nvalid;  // [modules]
  const uint16_t* W;        // [V, d] bf16
  const uint16_t* gamma;    // [d]
  const uint16_t* hidden[kMaxModules];
  uint16_t* dhidden[kMaxModules];
  float* loss_tok;          // [M] or null
  float* row_loss;          // [M]: token loss (0 when masked), for the module means
  int32_t* n_valid;         // [modules]
  float* loss_mean;         // [modules]
  uint32_t* flags;
};

// Largest width the on-chip backward handles: 8 CTAs of 256 columns.
constexpr int kFlashMaxD = 2048;
// CTAs per cluster (1, 2, 4 or 8) and d-columns per CTA (a multiple of 64) for width d.
int flash_cluster_size(int d);
int flash_slice_width(int d);
cudaError_t flash_prepare(int device);
// Kept-token counts and 1/Nvalid of the auxiliary modules (and bad-target flags).
cudaError_t launch_flash_count(const FlashArgs& a, float* inv_nvalid, cudaStream_t s);
// The on-chip forward + backward of the auxiliary rows; w: tensor map of W
// (bf16 [V, d], boxes of 64 columns x 64 rows, 128-byte swizzle).
cudaError_t launch_flash(const CUtensorMap& w, const FlashArgs& a, int device, int sms,
                         cudaStream_t s);
// Module means of the auxiliary modules from row_loss, in a fixed order.
cudaError_t launch_flash_means(const FlashArgs& a, cudaStream_t s);

// ---- row kernels ---------------------------------------------------------------

struct RowArgs {
  const uint16_t* hidden[kMaxModules];
  uint16_t* dhidden[kMaxModules];
  int64_t N;
  int32_t K;
  int32_t d;
  int32_t V;
  int32_t ldp;          // row stride (elements) of the exponential / gradient buffer
  int32_t n_tiles_v;    // column tiles of the logits product
  int32_t ignore_index;
  float eps;
  const uint16_t* gamma;
  const int32_t* targets;
  const uint8_t* mask;
  float* r;             // [M]
  uint16_t* xhat;       // [M, d]
  float* lse;           // [M]
  float* zy;            // [M]
  float* edz;           // [M]: E_p[s] - s_y per kept token (0 if masked), for the
                        //      RMSNorm backward's row sum
  float* nll;           // [M]: lse - z_y of a row whose target is in range (the
                        //      gradient's p_y - 1 = expm1(-nll) keeps its precision)
  float2* stats;        // [n_tiles_v, M]
  double* part_sum;     // [K, part_blocks]
  int32_t* part_cnt;    // [K, part_blocks]
  int32_t part_blocks;
  float* inv_nvalid;    // [K]
  float* loss_tok;      // [K, N] or null
  float* loss_mean;     // [K]
  uint16_t* P;          // [M, ldp] bf16: exp(z - tile max), turned into G in place
  float* dgamma_part;   // [dg_chunks, d]: per 32-row block of the final module
  int32_t dg_chunks;
  float* dgamma;        // [d] or null
  uint32_t* flags;
  // exit readout
  int32_t* argmax;       // [n_tiles_v, M]: first column of each tile's maximum
  int32_t* top1;         // [M] or null: first argmax over the vocabulary
  float* top1_logprob;   // [M] or null: log p of that entry
  // heads' temperature and bias
  const float* tau;      // [K] or null
  float* usum;           // [n_tiles_v, M] (with tau gradients)
  float* sy;             // [M]
  double* part_tau;      // [K, part_blocks]
  float* dtau;           // [K] or null
  float* dbias;          // [K, V] or null
  float* db_part;        // [K, db_chunks, ldp]
  int32_t db_chunks;     // row chunks per module of the bias-gradient pass
  // Rows whose gradient is the stored exponentials times per-row factors (the
  // log-sum-exp pass decides): row_fa = e^{-lse}, and row_fb = 1 - p_y for an
  // auxiliary row (the dX̂ epilogue's W_y term) or 0 for a final-module row
  // (its target entry and x̂ row are rewritten instead).  row_fa = -1 for the
  // rows the gradient pass turns into G (a tile stored against its own
  // maximum, or lse above 60).  Null: every row goes through the gradient pass.
  float* row_fa;         // [M]
  float* row_fb;         // [M]
  // Compaction of the kept tokens (null kept_local: every token keeps its row).
  // Kept tokens take rows [0, Mk) of the per-row buffers in token order, module
  // by module; each masked token zeroes one row of [Mk, M).
  int32_t* kept_local;   // [M] kept tokens before this one within its chunk of kScanRows
  int32_t* chunk_base;   // [K * nchunks] kept tokens before the chunk (counts, then prefix)
  int32_t nchunks;       // chunks of kScanRows tokens per module
  int32_t* offsets;      // [K + 1] first compact row of each module; offsets[K] = Mk
  int32_t* orig_row;     // [M] compact row -> token row k * N + n
  int32_t* tgt_c;        // [M] target of a compact row
  int32_t* grad_list;    // [M]: rows whose gradient pass takes the whole row
  int32_t* grad_count;   // [1]: their number (zeroed by the kept-token scan)
  int32_t grad_ctas;     // CTAs of the whole-row pass (a few per SM)
};

constexpr int kScanRows = 1024;  // tokens per block of the kept-token scan

constexpr int kGradRows = 128;   // rows per CTA of the bias-gradient pass

// Kept-token scan (with a.kept_local): per-chunk counts and in-chunk ranks,
// then the prefix over chunks and the modules' compact offsets.
cudaError_t launch_keep_scan(const RowArgs& a, cudaStream_t s);
cudaError_t launch_rmsnorm_fwd(const RowArgs& a, cudaStream_t s);
// heads: with the heads' temperature gradient (a.dtau) as well
cudaError_t launch_lse(const RowArgs& a, cudaStream_t s, bool heads = false);
// The exit readout's combine: log-sum-exp, top-1, and (with targets) losses.
cudaError_t launch_exit_lse(const RowArgs& a, cudaStream_t s);
// G in place; with a.dbias also the per-module column sums of dL/dz.
cudaError_t launch_grad(const RowArgs& a, cudaStream_t s);
cudaError_t launch_dgamma_reduce(const RowArgs& a, cudaStream_t s);

}  // namespace solo
