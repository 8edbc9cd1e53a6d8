// kvshot_api.cu -- host side of libkvshot's C ABI: argument validation, the
// work planner (kernel choice, row blocks, persistent grid, workspace
// layout), TMA tensor-map encoding and the launches.  No host synchronisation,
// no allocation.
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <mutex>

#include "kvshot_internal.h"

namespace kvshot {

// Defined in the kernel translation units.
cudaError_t attn_cc_occupancy(int C, int* ctas_per_sm);
cudaError_t attn_mma_occupancy(int m_tiles, int C, bool fp8, int* ctas_per_sm);
cudaError_t attn_tc_occupancy(int C, int* ctas_per_sm);

namespace {

constexpr int kVersion = 100;  // 0.1.0

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D view [rows, 128] of a bf16 tensor, boxes of {64 dims, box_rows rows},
// 128-byte swizzle (matches tile_off in kvshot_attn_common.cuh).
bool encode_rows(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(kHeadDim) * 2};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp8 E4M3 target cache: one byte per element, whole 128-byte rows per box, under the 128-byte
// swizzle (the m16n8k16 kernel decodes the codes from shared memory straight into MMA fragments).
bool encode_rows_fp8(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(kHeadDim)};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kHeadDim), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Grouped views of a [rows, 128] bf16 matrix for the tensor-memory kernel (kGroupBytes in
// kvshot_internal.h): a box lands as 8-row groups of 2 KB, each holding its rows' dims 0..63
// (128-byte swizzled) and then dims 64..127.
//  - 4-D {64 dims, 8 rows, 2 halves, rows / 8} (rows % 8 == 0), box {64, 8, 2, groups}: whole
//    8-row groups from a row-group coordinate (pages and aligned cache slices);
//  - 3-D {64 dims, rows, 2 halves}, box {64, 8, 2}: one group from any first row (draft slots).
// The halves dimension's stride (128 B) is below the rows' (256 B): both views address every
// element of the matrix exactly once.
bool encode_rows_grouped(CUtensorMap* map, const void* base, uint64_t rows, uint32_t groups) {
  auto fn = encode_fn();
  if (fn == nullptr || rows % 8 != 0) return false;
  const cuuint64_t dims[4] = {64, 8, 2, static_cast<cuuint64_t>(rows / 8)};
  const cuuint64_t strides[3] = {256, 128, 2048};
  const cuuint32_t box[4] = {64, 8, 2, groups};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_rows_group3(CUtensorMap* map, const void* base, uint64_t rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {64, static_cast<cuuint64_t>(rows), 2};
  const cuuint64_t strides[2] = {256, 128};
  const cuuint32_t box[3] = {64, 8, 2};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr int kMaxScaleExp = 64;

enum class Kernel { kCudaCore, kMma, kTensorMemory };

// Fixed cost, in 64-key tile times of one CTA, of splitting units across CTAs (piece epilogues
// that stall the pipeline mid-stream, the merge kernel after the last CTA); measured on GB300.
constexpr int64_t kSplitCostTiles = 15;

// Fewest 64-key tiles per CTA on an automatic grid: a CTA's prologue and every extra piece to merge
// cost more than the parallelism of one-tile CTAs brings on small, L2-resident problems (GB300:
// KV-only chain, 8 units of 33 tiles, m16n8k16 21.4 us per call on 264 CTAs against 14.4 us on 88,
// tcgen05 whole chain 21.4 against 17.3 us on 88; tiny chain, 8 units of 3 tiles, 11.8 against
// 10.5 us on 8 CTAs; 2, 4, 6 or 8 tiles per CTA measured slower).  Large problems have hundreds of
// tiles per CTA.
constexpr int64_t kMinTilesPerCta = 3;

}  // namespace

bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint32_t box_cols,
                    uint32_t box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

// 4-D view {128 dims, hq, Nq, C} of q [C, Nq, hq, 128]; a box is one 64-dim
// half of `heads` heads of one KV group for `nodes` draft nodes (rows node-major).
bool encode_q(CUtensorMap* map, const void* q, int C, int Nq, int hq, QBox qb) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[4] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(hq),
                              static_cast<cuuint64_t>(Nq), static_cast<cuuint64_t>(C)};
  const cuuint64_t row = static_cast<cuuint64_t>(kHeadDim) * 2;
  const cuuint64_t strides[3] = {row, row * hq, row * hq * Nq};
  const cuuint32_t box[4] = {64, static_cast<cuuint32_t>(qb.heads), static_cast<cuuint32_t>(qb.nodes), 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(q), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Plan {
  Kernel kernel;
  bool mma;
  int m_tiles;        // mma path
  int nq_box;         // tensor-memory path: draft nodes per 128-row block
  bool spread;        // tensor-memory path: 16 rows per TMEM lane quarter
  bool pair;          // tensor-memory path: two 128-row blocks per unit (stacks of more than 128 rows)
  int rows_per_unit;
  int row_blocks;
  int units;
  int num_ctas;
  int len_bound;
  int draft_tiles;
  size_t off_lse, off_o, bytes;
};

int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64 && cached[dev] > 0) return cached[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64) cached[dev] = n;
  return n;
}

// Checks that do not depend on the cache layout.
kvshot_status check_common(const kvshot_attn_desc* d) {
  if (d == nullptr) return KVSHOT_ERR_NULL;
  if (d->num_caches < 1 || d->num_seqs < 1 || d->num_caches % d->num_seqs != 0) return KVSHOT_ERR_SHAPE;
  if (d->num_caches > kMaxCaches) return KVSHOT_ERR_UNSUPPORTED;
  if (d->hq < 1 || d->hkv < 1 || d->hq % d->hkv != 0) return KVSHOT_ERR_SHAPE;
  if (d->head_dim != kHeadDim) return KVSHOT_ERR_UNSUPPORTED;
  if (d->n_nodes < 0 || d->n_query < 0 || d->n_query > d->n_nodes || d->n_nodes > d->n_max) return KVSHOT_ERR_SHAPE;
  if (d->max_seq_len < 0) return KVSHOT_ERR_SHAPE;
  if (!std::isfinite(d->scale) || d->scale < 0.f) return KVSHOT_ERR_SHAPE;  // the kernels fold a positive scale
  const uint32_t known =
      KVSHOT_TREE | KVSHOT_FORCE_CC | KVSHOT_FORCE_MMA | KVSHOT_FORCE_TC | KVSHOT_OVERLAP_PREVIOUS | KVSHOT_TARGET_FP8;
  if ((d->flags & ~known) != 0) return KVSHOT_ERR_SHAPE;
  if (d->flags & KVSHOT_TARGET_FP8) {
    if (d->k_scale_exp < -kMaxScaleExp || d->k_scale_exp > kMaxScaleExp || d->v_scale_exp < -kMaxScaleExp ||
        d->v_scale_exp > kMaxScaleExp)
      return KVSHOT_ERR_SHAPE;
    if (d->flags & KVSHOT_FORCE_CC) return KVSHOT_ERR_UNSUPPORTED;
    // The tensor-memory kernel decodes fp8 tiles for stacks of up to 128 rows (not for paired blocks).
    if ((d->flags & KVSHOT_FORCE_TC) && static_cast<int64_t>(d->hq / std::max(d->hkv, 1)) * d->n_query > 128)
      return KVSHOT_ERR_UNSUPPORTED;
  }
  const uint32_t force = d->flags & (KVSHOT_FORCE_CC | KVSHOT_FORCE_MMA | KVSHOT_FORCE_TC);
  if (force & (force - 1)) return KVSHOT_ERR_SHAPE;  // at most one kernel may be forced
  const int G = d->hq / d->hkv;
  if ((d->flags & KVSHOT_FORCE_TC) && (G > 128 || 128 % G != 0)) return KVSHOT_ERR_UNSUPPORTED;
  if ((d->flags & KVSHOT_TREE) && d->n_nodes > kMaxTreeNodes) return KVSHOT_ERR_UNSUPPORTED;
  if (d->num_ctas < 0) return KVSHOT_ERR_SHAPE;
  if (static_cast<int64_t>(d->num_caches) * d->hkv * d->n_max >= INT_MAX) return KVSHOT_ERR_UNSUPPORTED;
  return KVSHOT_OK;
}

kvshot_status check_attn_desc(const kvshot_attn_desc* d, bool paged) {
  if (kvshot_status st = check_common(d)) return st;
  if (paged) {
    // A 64-key tile must cover whole pages or lie inside one page: P in {8, 16, 32, 64, 128, 192, 256}.
    const int P = d->page_size;
    if (P < 8 || P > 256 || !(kTileKeys % P == 0 || P % kTileKeys == 0)) return KVSHOT_ERR_UNSUPPORTED;
    if (d->max_pages_per_seq < 1 || d->num_pages < 1) return KVSHOT_ERR_SHAPE;
    const int64_t rows = static_cast<int64_t>(d->num_pages) * d->hkv * d->page_size;
    if (rows >= INT_MAX) return KVSHOT_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(d->num_caches) * d->max_pages_per_seq >= INT_MAX) return KVSHOT_ERR_UNSUPPORTED;
  } else {
    if (d->l_cap < 1) return KVSHOT_ERR_SHAPE;
    if (static_cast<int64_t>(d->num_caches) * d->hkv * d->l_cap >= INT_MAX) return KVSHOT_ERR_UNSUPPORTED;
  }
  return KVSHOT_OK;
}

kvshot_status make_plan(const kvshot_attn_desc* d, bool paged, Plan* pl) {
  const int G = d->hq / d->hkv;
  const int rows = G * d->n_query;
  const bool force_cc = d->flags & KVSHOT_FORCE_CC, force_tc = d->flags & KVSHOT_FORCE_TC;
  const bool force_mma = d->flags & KVSHOT_FORCE_MMA;
  // Kernel choice, measured on GB300 (bench + ncu):
  //  - below 16 stacked rows per KV head the m16n8k16 kernel streams K/V at
  //    90-94% of HBM bandwidth (4 rows: 187 us per ragged-chain call against
  //    202 us for the tcgen05 kernel), also where the CUDA-core kernel is issue
  //    bound (IPC ~1, ~100 warp instructions per key, 23%); the CUDA-core
  //    kernel stays behind KVSHOT_FORCE_CC;
  //  - from 16 rows on, the tcgen05 kernel, whose MMAs run asynchronously out
  //    of shared memory into tensor memory, is faster: 314 us against 323 us
  //    per multi-layer-tree call at 16 rows (spread rows), 1.9x at 48 rows,
  //    3-4x for whole-tree stacks of 128-256 rows.
  const bool tc_ok = G <= 128 && 128 % G == 0;
  // fp8 tiles: both kernels decode them (the tensor-memory kernel for stacks of up to 128 rows).  The
  // producer warps' decode into shared memory for the tcgen05 MMAs is the faster path for 17-128 rows
  // (hybrid tree per depth, 32-48 rows: 85 us against 103 us per call for the m16n8k16 kernel, which
  // decodes in registers); at 16 rows and below the m16n8k16 kernel is far ahead (264 us against 476 us).
  const bool fp8 = d->flags & KVSHOT_TARGET_FP8;
  const bool tc_auto = fp8 ? (rows > 16 && rows <= 128) : rows >= 16;
  const Kernel automatic = (tc_auto && tc_ok) ? Kernel::kTensorMemory : Kernel::kMma;
  pl->kernel = force_cc ? Kernel::kCudaCore : force_tc ? Kernel::kTensorMemory
                                           : force_mma ? Kernel::kMma : automatic;
  pl->mma = pl->kernel == Kernel::kMma;
  pl->m_tiles = 0;
  pl->nq_box = 0;
  pl->spread = false;
  pl->pair = false;
  if (pl->kernel == Kernel::kMma) {
    pl->m_tiles = std::min(kMmaMaxTiles, std::max(1, (rows + 15) / 16));
    pl->rows_per_unit = 16 * pl->m_tiles;
  } else if (pl->kernel == Kernel::kTensorMemory) {
    pl->nq_box = std::max(1, std::min(d->n_query, 128 / G));
    pl->rows_per_unit = G * pl->nq_box;
    pl->spread = pl->rows_per_unit <= kSpreadMaxRows;
    // More than 128 rows: each unit takes two 128-row blocks, so every K/V tile feeds both.
    pl->pair = rows > 128;
    if (pl->pair) pl->rows_per_unit = 2 * 128;
  } else {
    pl->rows_per_unit = kCcRows;
  }
  pl->row_blocks = std::max(1, (rows + pl->rows_per_unit - 1) / pl->rows_per_unit);
  const int64_t units = static_cast<int64_t>(d->num_caches) * d->hkv * pl->row_blocks;
  const int64_t cap = paged ? static_cast<int64_t>(d->max_pages_per_seq) * d->page_size : d->l_cap;
  pl->len_bound = static_cast<int>(std::min<int64_t>(d->max_seq_len, cap));
  pl->draft_tiles = (d->n_nodes + kTileKeys - 1) / kTileKeys;
  // Upper bound on the tiles of any call with this descriptor (independent of the layout, so the
  // workspace size query and the call agree).
  const int64_t max_tiles =
      units * ((static_cast<int64_t>(d->max_seq_len) + kTileKeys - 1) / kTileKeys + pl->draft_tiles);
  if (units >= INT_MAX / 2 || max_tiles >= INT_MAX / 2) return KVSHOT_ERR_UNSUPPORTED;
  pl->units = static_cast<int>(units);
  int grid = d->num_ctas;
  if (grid == 0) {
    int per_sm = 0;
    const cudaError_t e = pl->kernel == Kernel::kMma ? attn_mma_occupancy(pl->m_tiles, d->num_caches, fp8, &per_sm)
                          : pl->kernel == Kernel::kTensorMemory ? attn_tc_occupancy(d->num_caches, &per_sm)
                                                                 : attn_cc_occupancy(d->num_caches, &per_sm);
    const int sms = sm_count();
    if (e != cudaSuccess || per_sm < 1 || sms < 1) return KVSHOT_ERR_CUDA;
    grid = sms * per_sm;
    // Tensor-memory kernel: when every unit fits on a CTA of its own and the SMs that would stay
    // idle would take fewer than kSplitCostTiles tiles off each CTA, give each unit its own CTA:
    // no unit is split, so no piece epilogue runs mid-stream and the merge has nothing to do.
    // (GB300, 128 units of 65 tiles, 16-token pages: 56.4 us per call on 128 CTAs against 59.9 us
    // on 152; 128 units of 514 tiles stay faster split over all SMs.)
    if (pl->kernel == Kernel::kTensorMemory && units <= grid) {
      const int64_t unit_tiles = (static_cast<int64_t>(d->max_seq_len) + kTileKeys - 1) / kTileKeys + pl->draft_tiles;
      if (unit_tiles * (grid - units) < kSplitCostTiles * static_cast<int64_t>(grid)) grid = static_cast<int>(units);
    }
  }
  if (d->num_ctas == 0)
    grid = static_cast<int>(std::min<int64_t>(grid, (max_tiles + kMinTilesPerCta - 1) / kMinTilesPerCta));
  grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(grid, std::max<int64_t>(1, max_tiles))));
  pl->num_ctas = grid;
  const size_t slots = static_cast<size_t>(pl->units) + grid;
  pl->off_lse = 0;
  pl->off_o = pl->off_lse + round_up(sizeof(float) * slots * pl->rows_per_unit, 256);
  pl->bytes = pl->off_o + sizeof(float) * slots * pl->rows_per_unit * kHeadDim;
  return KVSHOT_OK;
}

}  // namespace
}  // namespace kvshot

using namespace kvshot;

extern "C" const char* kvshot_status_string(kvshot_status s) {
  switch (s) {
    case KVSHOT_OK: return "ok";
    case KVSHOT_ERR_NULL: return "a required pointer is NULL";
    case KVSHOT_ERR_SHAPE: return "inconsistent or out-of-range sizes";
    case KVSHOT_ERR_ALIGN: return "misaligned pointer";
    case KVSHOT_ERR_UNSUPPORTED: return "valid but unsupported by this build";
    case KVSHOT_ERR_TREE: return "tree_parent entry is not an earlier node or -1";
    case KVSHOT_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case KVSHOT_ERR_CUDA: return "CUDA call failed";
    case KVSHOT_ERR_DEVICE_BOUNDS: return "page id or sequence length out of bounds";
    case KVSHOT_ERR_TIMEOUT: return "device pipeline wait timed out";
  }
  return "unknown status";
}

extern "C" int32_t kvshot_version(void) { return kVersion; }

extern "C" size_t kvshot_draft_attn_workspace_size(const kvshot_attn_desc* d) {
  if (d == nullptr || check_common(d) != KVSHOT_OK) return 0;
  if (d->n_query == 0) return 256;
  Plan pl;
  if (make_plan(d, false, &pl) != KVSHOT_OK) return 0;  // the size does not depend on the layout
  return pl.bytes;
}

extern "C" kvshot_status kvshot_draft_attn(const kvshot_attn_desc* d, const void* q, const void* target_k,
                                           const void* target_v, const int32_t* page_table,
                                           const int32_t* seq_lens, const void* draft_k, const void* draft_v,
                                           const int32_t* tree_parent, void* out, float* lse,
                                           kvshot_stream_t stream) {
  const bool paged = page_table != nullptr;
  if (kvshot_status st = check_attn_desc(d, paged)) return st;
  if (d->n_query == 0) return KVSHOT_OK;
  const bool tree = d->flags & KVSHOT_TREE;
  if (!q || !target_k || !target_v || !seq_lens || !draft_k || !draft_v || !out || !lse) return KVSHOT_ERR_NULL;
  if (tree && !tree_parent) return KVSHOT_ERR_NULL;
  if (!aligned(q, 16) || !aligned(target_k, 16) || !aligned(target_v, 16) || !aligned(draft_k, 16) ||
      !aligned(draft_v, 16) || !aligned(out, 16) || !aligned(lse, 4) || !aligned(seq_lens, 4) ||
      (paged && !aligned(page_table, 4)) || (tree && !aligned(tree_parent, 4)))
    return KVSHOT_ERR_ALIGN;
  Plan pl;
  if (kvshot_status st = make_plan(d, paged, &pl)) return st;
  if (d->workspace == nullptr || !aligned(d->workspace, 256) || d->workspace_bytes < pl.bytes)
    return KVSHOT_ERR_WORKSPACE;

  TensorMaps maps;
  const uint64_t trows = paged ? static_cast<uint64_t>(d->num_pages) * d->hkv * d->page_size
                               : static_cast<uint64_t>(d->num_caches) * d->hkv * d->l_cap;
  const uint32_t tbox = paged ? static_cast<uint32_t>(std::min(d->page_size, kTileKeys)) : kTileKeys;
  const uint64_t drows = static_cast<uint64_t>(d->num_caches) * d->hkv * d->n_max;
  const bool fp8 = (d->flags & KVSHOT_TARGET_FP8) != 0;
  // The tensor-memory kernel stages tiles in the grouped layout: target tiles whenever their rows
  // start on a multiple of 8 (always when paged; contiguous caches with l_cap % 8 == 0), draft tiles always.
  const bool tmem_kernel = pl.kernel == Kernel::kTensorMemory;
  // (fp8 prefix tiles are decoded into the grouped layout whatever the cache layout.)  The m16n8k16
  // kernel stages every tile of a bf16 paged cache grouped too (prefix_grouped then covers its draft
  // tiles): one box per page with both halves halves the TMA boxes a tile takes, which bounds small
  // pages (GB300, ragged chain of 64 caches: 8-token pages 0.75 -> 0.92 of the copy peak, 16-token
  // pages 0.93 -> 0.94).
  const bool prefix_grouped =
      tmem_kernel ? (fp8 || paged || d->l_cap % 8 == 0) : (pl.kernel == Kernel::kMma && paged && !fp8);
  bool tmaps;
  if (fp8) {
    tmaps = encode_rows_fp8(&maps.tk, target_k, trows, tbox) && encode_rows_fp8(&maps.tv, target_v, trows, tbox);
  } else if (prefix_grouped) {
    const uint32_t groups = (paged ? std::min(d->page_size, kTileKeys) : kTileKeys) / 8;
    tmaps = encode_rows_grouped(&maps.tk, target_k, trows, groups) &&
            encode_rows_grouped(&maps.tv, target_v, trows, groups);
  } else {
    tmaps = encode_rows(&maps.tk, target_k, trows, tbox) && encode_rows(&maps.tv, target_v, trows, tbox);
  }
  const bool dmaps = tmem_kernel || prefix_grouped ? encode_rows_group3(&maps.dk, draft_k, drows) &&
                                       encode_rows_group3(&maps.dv, draft_v, drows)
                                 : encode_rows(&maps.dk, draft_k, drows, kDraftBoxRows) &&
                                       encode_rows(&maps.dv, draft_v, drows, kDraftBoxRows);
  if (!tmaps || !dmaps) return KVSHOT_ERR_CUDA;
  if (tmem_kernel) {
    if (!encode_q(&maps.q, q, d->num_caches, d->n_query, d->hq, q_box(d->hq / d->hkv, pl.nq_box, pl.spread)))
      return KVSHOT_ERR_CUDA;
  } else {
    maps.q = maps.tk;  // unused by the other kernels
  }

  AttnParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.out = static_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  p.page_table = page_table;
  p.seq_lens = seq_lens;
  p.tree_parent = tree_parent;
  p.err = d->err_flag;
  uint8_t* ws = static_cast<uint8_t*>(d->workspace);
  p.ws_lse = reinterpret_cast<float*>(ws + pl.off_lse);
  p.ws_o = reinterpret_cast<float*>(ws + pl.off_o);
  p.C = d->num_caches;
  p.B = d->num_seqs;
  p.hq = d->hq;
  p.hkv = d->hkv;
  p.G = d->hq / d->hkv;
  p.rows_total = p.G * d->n_query;
  p.rows_per_unit = pl.rows_per_unit;
  p.row_blocks = pl.row_blocks;
  p.paged = paged ? 1 : 0;
  p.page_size = paged ? d->page_size : kTileKeys;
  p.max_pages = paged ? d->max_pages_per_seq : 0;
  p.num_pages = paged ? d->num_pages : 0;
  p.l_cap = paged ? 0 : d->l_cap;
  p.box_rows = static_cast<int>(tbox);
  p.len_bound = pl.len_bound;
  p.N = d->n_nodes;
  p.Nq = d->n_query;
  p.n_max = d->n_max;
  p.tree = tree ? 1 : 0;
  p.draft_tiles = pl.draft_tiles;
  const double scale = d->scale != 0.f ? static_cast<double>(d->scale) : 1.0 / std::sqrt(static_cast<double>(kHeadDim));
  p.qscale = static_cast<float>(scale * 1.4426950408889634);
  p.num_ctas = pl.num_ctas;
  p.fp8 = fp8 ? 1 : 0;
  p.prefix_grouped = prefix_grouped ? 1 : 0;
  p.wait_ns = d->wait_limit_ns != 0 ? d->wait_limit_ns : static_cast<uint32_t>(2000000000u);
  p.k_scale = fp8 ? std::ldexp(1.f, d->k_scale_exp) : 1.f;
  p.v_scale = fp8 ? std::ldexp(1.f, d->v_scale_exp) : 1.f;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const bool pdl = (d->flags & KVSHOT_OVERLAP_PREVIOUS) != 0;
  cudaError_t e = pl.kernel == Kernel::kMma            ? launch_attn_mma(p, maps, pl.m_tiles, pdl, s)
                  : pl.kernel == Kernel::kTensorMemory ? launch_attn_tc(p, maps, pl.nq_box, pl.spread, pl.pair, pdl, s)
                                                       : launch_attn_cc(p, maps, pdl, s);
  if (e != cudaSuccess) return KVSHOT_ERR_CUDA;
  e = launch_merge(p, s);
  return e == cudaSuccess ? KVSHOT_OK : KVSHOT_ERR_CUDA;
}

namespace {

kvshot_status draft_append(const kvshot_attn_desc* d, const void* q_in, const void* k_in, const void* v_in,
                           const int32_t* positions, int32_t n0, int32_t n_new, float rope_base, const void* q_norm_w,
                           const void* k_norm_w, float eps, void* draft_k, void* draft_v, void* q_out,
                           kvshot_stream_t stream) {
  if (d == nullptr) return KVSHOT_ERR_NULL;
  if (d->num_caches < 1 || d->hq < 1 || d->hkv < 1 || d->n_max < 0) return KVSHOT_ERR_SHAPE;
  if (d->head_dim != kHeadDim) return KVSHOT_ERR_UNSUPPORTED;
  if (n0 < 0 || n_new < 0 || static_cast<int64_t>(n0) + n_new > d->n_max) return KVSHOT_ERR_SHAPE;
  if (!(rope_base > 0.f) || !std::isfinite(rope_base)) return KVSHOT_ERR_SHAPE;
  if (n_new == 0) return KVSHOT_OK;
  if (static_cast<int64_t>(d->num_caches) * n_new >= INT_MAX ||
      static_cast<int64_t>(d->num_caches) * d->hkv * d->n_max >= INT_MAX)
    return KVSHOT_ERR_UNSUPPORTED;
  if (!q_in || !k_in || !v_in || !positions || !draft_k || !draft_v || !q_out) return KVSHOT_ERR_NULL;
  if (!aligned(q_in, 16) || !aligned(k_in, 16) || !aligned(v_in, 16) || !aligned(draft_k, 16) ||
      !aligned(draft_v, 16) || !aligned(q_out, 16) || !aligned(positions, 4))
    return KVSHOT_ERR_ALIGN;
  // q_out may be q_in exactly, but must not partially overlap it.
  const size_t qbytes = static_cast<size_t>(d->num_caches) * n_new * d->hq * kHeadDim * 2;
  const uintptr_t a = reinterpret_cast<uintptr_t>(q_in), b = reinterpret_cast<uintptr_t>(q_out);
  if (a != b && a < b + qbytes && b < a + qbytes) return KVSHOT_ERR_SHAPE;
  AppendParams ap;
  ap.q_in = static_cast<const __nv_bfloat16*>(q_in);
  ap.k_in = static_cast<const __nv_bfloat16*>(k_in);
  ap.v_in = static_cast<const __nv_bfloat16*>(v_in);
  ap.positions = positions;
  ap.draft_k = static_cast<__nv_bfloat16*>(draft_k);
  ap.draft_v = static_cast<__nv_bfloat16*>(draft_v);
  ap.q_out = static_cast<__nv_bfloat16*>(q_out);
  ap.C = d->num_caches;
  ap.hq = d->hq;
  ap.hkv = d->hkv;
  ap.n_max = d->n_max;
  ap.n0 = n0;
  ap.n_new = n_new;
  for (int j = 0; j < kHeadDim / 2; ++j)
    ap.inv_freq[j] = std::pow(static_cast<double>(rope_base), -2.0 * j / kHeadDim);
  ap.q_norm_w = static_cast<const __nv_bfloat16*>(q_norm_w);
  ap.k_norm_w = static_cast<const __nv_bfloat16*>(k_norm_w);
  ap.eps = eps;
  const cudaError_t e = launch_append(ap, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? KVSHOT_OK : KVSHOT_ERR_CUDA;
}

}  // namespace

extern "C" kvshot_status kvshot_draft_append(const kvshot_attn_desc* d, const void* q_in, const void* k_in,
                                             const void* v_in, const int32_t* positions, int32_t n0,
                                             int32_t n_new, float rope_base, void* draft_k, void* draft_v,
                                             void* q_out, kvshot_stream_t stream) {
  return draft_append(d, q_in, k_in, v_in, positions, n0, n_new, rope_base, nullptr, nullptr, 0.f, draft_k, draft_v,
                      q_out, stream);
}

extern "C" kvshot_status kvshot_draft_append_qknorm(const kvshot_attn_desc* d, const void* q_in, const void* k_in,
                                                    const void* v_in, const int32_t* positions, int32_t n0,
                                                    int32_t n_new, float rope_base, const void* q_norm_w,
                                                    const void* k_norm_w, float eps, void* draft_k, void* draft_v,
                                                    void* q_out, kvshot_stream_t stream) {
  if (d == nullptr) return KVSHOT_ERR_NULL;
  if (!(eps > 0.f) || !std::isfinite(eps)) return KVSHOT_ERR_SHAPE;
  if (n_new > 0 && (q_norm_w == nullptr || k_norm_w == nullptr)) return KVSHOT_ERR_NULL;
  if (!aligned(q_norm_w, 4) || !aligned(k_norm_w, 4)) return KVSHOT_ERR_ALIGN;
  return draft_append(d, q_in, k_in, v_in, positions, n0, n_new, rope_base, q_norm_w, k_norm_w, eps, draft_k, draft_v,
                      q_out, stream);
}
