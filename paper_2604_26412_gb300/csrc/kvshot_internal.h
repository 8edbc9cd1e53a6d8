// kvshot_internal.h -- declarations shared by libkvshot's translation units.
//
// Work decomposition of kvshot_draft_attn (see kvshot_attn_common.cuh):
//   unit  = (cache c, KV head h, row block rb): the stacked query rows of one
//           GQA group (G heads x Nq draft nodes, or a 64-row block of them).
//           Every unit streams the same keys: L_c prefix tokens then the N
//           draft slots.
//   tile  = TK consecutive keys of one unit (prefix tiles first, then draft
//           tiles), staged into shared memory by TMA as one K and one V block.
//   The tiles of all units are laid end to end (cache-major) and cut into
//   equal contiguous ranges, one per persistent CTA ("stream-K" split), so
//   ragged prefix lengths stay balanced.  A unit whose tiles straddle CTAs is
//   computed as pieces whose softmax states are merged afterwards.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kvshot.h"

namespace kvshot {

constexpr int kHeadDim = 128;
constexpr int kTileKeys = 64;                         // TK
constexpr int kHalfBytes = kTileKeys * 128;           // 64 dims x TK keys, bf16: one TMA-swizzled half
constexpr int kKVTileBytes = 2 * kHalfBytes;          // one K (or V) tile
constexpr int kStageBytes = 2 * kKVTileBytes;         // K + V
constexpr int kMaxCaches = 1024;
constexpr int kMaxTreeNodes = 64;
constexpr int kDraftBoxRows = 8;                      // draft K/V are loaded 8 rows per TMA box
constexpr int kCcRows = 4;                            // rows per unit of the CUDA-core kernel
constexpr int kMmaMaxTiles = 4;                       // m16 tiles per unit of the tensor-core kernel
constexpr int kSpreadMaxRows = 64;                    // tensor-memory kernel: units up to this many rows are spread
// Grouped tile layout of the tensor-memory kernel: a K (or V) tile is 8 groups
// of 8 keys; group g starts at byte g * kGroupBytes and holds its keys' dims
// 0..63 (1 KB, 128-byte swizzled rows) then dims 64..127 (kGroupHalfBytes on).
// One TMA box then brings whole groups with both halves, e.g. a whole
// 16-token page in one 4 KB box.
constexpr int kGroupBytes = 8 * 256;
constexpr int kGroupHalfBytes = 8 * 128;

// Query box of the tensor-memory kernel's 4-D q map {128, hq, Nq, C}: `heads`
// heads of the KV group x `nodes` draft nodes.  Dense units load all G x nq_box
// stacked rows as one box.  Spread units (<= 64 rows) put 16 stacked rows in
// each 32-lane TMEM quarter, so a box holds at most 16 rows.
struct QBox {
  int heads, nodes;
};
__host__ __device__ inline QBox q_box(int G, int nq_box, bool spread) {
  if (!spread) return QBox{G, nq_box};
  if (G >= 16) return QBox{16, 1};
  return QBox{G, nq_box < 16 / G ? nq_box : 16 / G};
}

// Everything a draft-attention kernel needs besides the tensor maps.
struct AttnParams {
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* lse;
  const int32_t* page_table;
  const int32_t* seq_lens;
  const int32_t* tree_parent;
  int32_t* err;             // may be null
  float* ws_lse;            // [slots, rows_per_unit] log2-domain lse of pieces
  float* ws_o;              // [slots, rows_per_unit, 128] normalised piece outputs
  int C, B, hq, hkv, G;
  int rows_total;           // G * Nq
  int rows_per_unit;        // rows of one unit (<= rows_total)
  int row_blocks;           // RB = ceil(rows_total / rows_per_unit)
  int paged, page_size, max_pages, num_pages, l_cap;
  int box_rows;             // rows per target TMA box: min(page_size, TK) paged, TK contiguous
  int len_bound;            // min(max_seq_len, capacity): seq_lens are clamped to [0, len_bound]
  int N, Nq, n_max, tree;
  int draft_tiles;          // ceil(N / TK)
  float qscale;             // softmax scale * log2(e): scores are kept in the log2 domain
  int num_ctas;             // persistent grid size
  int fp8;                  // target K/V are e4m3 codes (KVSHOT_TARGET_FP8; m16n8k16 kernel only)
  int prefix_grouped;       // prefix tiles are staged in the grouped layout (tensor-memory kernel: draft tiles always;
                            // m16n8k16 kernel: draft tiles too)
  uint32_t wait_ns;         // limit on any one pipeline wait (desc->wait_limit_ns, default 2 s)
  float k_scale, v_scale;   // fp8: 2^k_scale_exp, 2^v_scale_exp
};

struct AppendParams {
  const __nv_bfloat16* q_in;
  const __nv_bfloat16* k_in;
  const __nv_bfloat16* v_in;
  const int32_t* positions;
  __nv_bfloat16* draft_k;
  __nv_bfloat16* draft_v;
  __nv_bfloat16* q_out;
  int C, hq, hkv, n_max, n0, n_new;
  double inv_freq[kHeadDim / 2];  // rope_base^(-2j/128) in fp64
  // QK-norm (kvshot_draft_append_qknorm): per-head RMSNorm weights over the 128 dims, or null.
  const __nv_bfloat16* q_norm_w;
  const __nv_bfloat16* k_norm_w;
  float eps;
};

// Target and draft K/V maps.  The m16n8k16 and CUDA-core kernels use 2-D
// maps (boxes of one 64-dim half); the tensor-memory kernel uses grouped maps
// (4-D target, 3-D draft: boxes of whole 8-key groups, both halves) except
// for a contiguous target cache whose l_cap is not a multiple of 8.
struct TensorMaps {
  CUtensorMap tk, tv, dk, dv;
  CUtensorMap q;  // [C, Nq, hq, 128] as 4-D {128, hq, Nq, C}; used by the tensor-memory kernel
};

// Encodes a 2-D tiled tensor map over a row-major bf16 matrix [rows, cols] (row pitch cols * 2
// bytes), boxes of {box_cols, box_rows}, 128-byte swizzle.  False if the encoder is unavailable
// or rejects the layout.
bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint32_t box_cols,
                    uint32_t box_rows);

// Kernel launchers (one per translation unit).  Return cudaSuccess or the launch error.  `pdl`:
// launch with programmatic stream serialization (KVSHOT_OVERLAP_PREVIOUS).
cudaError_t launch_attn_cc(const AttnParams& p, const TensorMaps& maps, bool pdl, cudaStream_t stream);
cudaError_t launch_attn_mma(const AttnParams& p, const TensorMaps& maps, int m_tiles, bool pdl, cudaStream_t stream);
cudaError_t launch_attn_tc(const AttnParams& p, const TensorMaps& maps, int nq_box, bool spread, bool pair, bool pdl,
                           cudaStream_t stream);

// Launches `kernel` on grid x block with `smem` dynamic bytes; with programmatic stream
// serialization when `pdl` is set.
template <typename... Args, typename... Actual>
cudaError_t launch_maybe_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, bool pdl,
                             cudaStream_t stream, Actual&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Actual&&>(args)...);
}
cudaError_t launch_merge(const AttnParams& p, cudaStream_t stream);
cudaError_t launch_append(const AppendParams& a, cudaStream_t stream);  // with QK-norm when a.q_norm_w is set

// CTAs per SM each kernel variant is built for (its shared-memory ring and
// register budget are sized for this residency).
int attn_cc_ctas_per_sm();
int attn_mma_ctas_per_sm(int m_tiles);

}  // namespace kvshot
