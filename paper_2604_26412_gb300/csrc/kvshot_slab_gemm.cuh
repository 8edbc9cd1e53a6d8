// kvshot_slab_gemm.cuh -- a table-driven tcgen05 GEMM that writes fp32
// "slabs": for each entry z of a small table, a weight matrix's 128-row block
// times a block of up to 128 token rows,
//   slab[z][t][f] = sum_k W_z[f][wx0 + k] * A_z[t][ax0 + k]          (one operand)
//   slab[z][t][f] = sum_k W_z[f][wx0 + k] * (A1_z[t][ax0 + k] - A0_z[t][ax0 + k])
//                                                                     (two operands)
// over k in [0, 64 nk).  A difference of bf16 activations is never formed or
// rounded: with at most 128 tokens per block, the two-operand form stacks
// A0's and A1's token rows in one B tile (one MMA of N = 2 x tokens) and
// subtracts the two fp32 products when it stores them; with more, it issues
// per 16-wide k step the MMA of W with A1 and then the MMA of W with A0 with
// the weight operand negated, both into one fp32 accumulator.  (The stacked
// form reads each weight tile from shared memory once instead of twice,
// which measured faster where it fits.)  Callers add the slabs they need and
// apply their epilogue in a kernel of their own.
//
// Shapes: A = 128 weight rows x 64 k (K-major, 128-byte swizzle, TMA box
// {64, 128}); B = up to 256 token rows x 64 k (box {64, box_tok}, MMA N =
// box_tok rounded up to 16); fp32 accumulators in TMEM.  Grid (token blocks
// of box_tok = min(T, 256), output-feature blocks of 128, table entries), the
// token block fastest so that a weight tile's token blocks run together and
// the weights leave HBM once.  128 threads: warp 0
// lane 0 issues the TMA loads, warp 1 owns TMEM and its lane 0 issues the
// MMAs, all four warps move the accumulators to the slab (thread = TMEM lane =
// output feature; a warp stores 32 consecutive features of one token).
#pragma once

#include "kvshot_attn_common.cuh"
#include "kvshot_tcgen05.cuh"

namespace kvshot {
namespace sg {
namespace {

using namespace dev;
using namespace tc;

constexpr int kFeat = 128;                  // output features per CTA (MMA M)
constexpr int kMaxTok = 256;                // tokens per CTA (MMA N)
constexpr int kKT = 64;                     // K per stage: one 128-byte swizzled row
constexpr int kMaxStages = 6;               // ring slots of 16 KB + (1 or 2) x N x 128 bytes
constexpr int kThreads = 128;
constexpr int kABytes = kFeat * kKT * 2;    // 16 KB
constexpr int kRingBytes = 192 * 1024;
constexpr uint32_t kTmemCols = 256;         // one accumulator of N <= 256 columns
constexpr uint32_t kNegateA = 1u << 13;     // instruction descriptor: negate the A (weight) operand
constexpr int kMaxEntries = 16;

struct Entry {
  int8_t w;    // weight map index
  int8_t a0;   // activation map index
  int8_t a1;   // second activation map index, or -1 (one operand)
  int8_t pad;
  int wx0;     // first weight column (element)
  int ax0;     // first activation column (element)
  int nk;      // k-tiles of 64
};

struct Params {
  Entry e[kMaxEntries];
  float* slab;   // [entries][T][d_out]
  int32_t* err;
  int T;         // token rows
  int d_out;     // output features (multiple of 128)
  int box_tok;   // token rows per TMA box and token block: min(T, 256)
};

// MMA N (and token-tile rows in shared memory) for a token block of box_tok rows.
__host__ __device__ inline int mma_n(int box_tok) { return (box_tok + 15) / 16 * 16; }

struct Maps {
  CUtensorMap w[2];  // weights [d_out, K], boxes {64, 128}
  CUtensorMap a[2];  // activations [T, K], boxes {64, box_tok}
};

inline size_t smem_bytes() { return 1024 + kRingBytes + 8 * (2 * kMaxStages + 1) + 16; }

// 2-D tiled TMA load with the default L2 policy (activations: every feature block reads them).
__device__ __forceinline__ void tma_load_2d_nohint(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__global__ void __launch_bounds__(kThreads, 1) slab_gemm(const __grid_constant__ Params p, const __grid_constant__ Maps maps) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();
  const int tt = blockIdx.x, ft = blockIdx.y, z = blockIdx.z;
  const Entry en = p.e[z];
  const bool both = en.a1 >= 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // Ring slot s: the weight tile at base + s * slot, the token tile(s) right after it.
  const int N = mma_n(p.box_tok);
  const int btile = N * kKT * 2;
  const bool stacked = both && 2 * N <= static_cast<int>(kTmemCols);  // [A0 rows; A1 rows]: N_mma = 2 N
  const int slot = kABytes + (both ? 2 : 1) * btile;
  const int nst = min(kMaxStages, kRingBytes / slot);
  uint64_t* full = reinterpret_cast<uint64_t*>(base + kRingBytes);
  uint64_t* empty = full + kMaxStages;
  uint64_t* done = empty + kMaxStages;
  uint32_t* tmem_base = reinterpret_cast<uint32_t*>(done + 1);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kMaxStages; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), 1);
    }
    mbar_init(smem_addr(done), 1);
    fence_mbar_init();
    prefetch_tensormap(&maps.w[en.w]);
    prefetch_tensormap(&maps.a[en.a0]);
    if (both) prefetch_tensormap(&maps.a[en.a1]);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base;
  const int nk = en.nk;
  bool ok = true;
  if (warp == 0 && lane == 0) {
    const uint64_t stream_once = l2_policy_evict_first();  // weights: read once
    const uint32_t tx = kABytes + (both ? 2 : 1) * p.box_tok * 128;
    const int ty = tt * p.box_tok;
    for (int kt = 0; kt < nk && ok; ++kt) {
      const int s = kt % nst;
      if (kt >= nst) ok = mbar_wait(smem_addr(&empty[s]), ((kt - nst) / nst) & 1, p.err);
      if (!ok) break;
      const uint32_t fb = smem_addr(&full[s]);
      mbar_arrive_expect_tx(fb, tx);
      tma_load_2d(smem_addr(base + s * slot), &maps.w[en.w], en.wx0 + kt * kKT, ft * kFeat, fb, stream_once);
      const uint32_t bdst = smem_addr(base + s * slot + kABytes);
      tma_load_2d_nohint(bdst, &maps.a[en.a0], en.ax0 + kt * kKT, ty, fb);
      if (both) tma_load_2d_nohint(bdst + btile, &maps.a[en.a1], en.ax0 + kt * kKT, ty, fb);
    }
  } else if (warp == 1 && lane == 0) {
    const uint32_t idesc = idesc_bf16(kFeat, stacked ? 2 * N : N, false);
    for (int kt = 0; kt < nk && ok; ++kt) {
      const int s = kt % nst;
      ok = mbar_wait(smem_addr(&full[s]), (kt / nst) & 1, p.err);
      if (!ok) break;
      tc_fence_after();
      const uint32_t a0 = smem_addr(base + s * slot), b0 = a0 + kABytes;
#pragma unroll
      for (int ks = 0; ks < kKT / 16; ++ks) {
        const uint64_t a = smem_desc_sw128(a0 + ks * 32, 16, 1024);
        if (both && !stacked) {  // + W A1, then - W A0
          tc_mma(tmem, a, smem_desc_sw128(b0 + btile + ks * 32, 16, 1024), idesc, (kt | ks) ? 1u : 0u);
          tc_mma(tmem, a, smem_desc_sw128(b0 + ks * 32, 16, 1024), idesc | kNegateA, 1u);
        } else {
          tc_mma(tmem, a, smem_desc_sw128(b0 + ks * 32, 16, 1024), idesc, (kt | ks) ? 1u : 0u);
        }
      }
      tc_commit(smem_addr(&empty[s]));
    }
    tc_commit(smem_addr(done));  // every MMA this thread issued has completed
  }
  __syncwarp();
  ok = mbar_wait(smem_addr(done), 0, p.err);
  tc_fence_after();
  const int f = ft * kFeat + warp * 32 + lane;
  const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  float* slab = p.slab + static_cast<size_t>(z) * p.T * p.d_out;
#pragma unroll 1
  for (int c = 0; c < N / 32 + (N % 32 != 0); ++c) {
    const int t0 = tt * p.box_tok + c * 32;
    const int nt = min(32, min(p.T, (tt + 1) * p.box_tok) - t0);
    if (nt <= 0) break;
    uint32_t x[32], y[32];
    tmem_ld32(trow + c * 32, x);
    if (stacked) tmem_ld32(trow + N + c * 32, y);
    tmem_wait_ld();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float v = stacked ? __uint_as_float(y[j]) - __uint_as_float(x[j]) : __uint_as_float(x[j]);
      if (j < nt) slab[static_cast<size_t>(t0 + j) * p.d_out + f] = ok ? v : 0.f;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// Launches slab_gemm over `entries` table entries.
inline cudaError_t launch(const Params& p, const Maps& maps, int entries, cudaStream_t stream) {
  const size_t smem = smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(slab_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const dim3 grid((p.T + p.box_tok - 1) / p.box_tok, p.d_out / kFeat, entries);
  slab_gemm<<<grid, kThreads, smem, stream>>>(p, maps);
  return cudaGetLastError();
}

}  // namespace
}  // namespace sg
}  // namespace kvshot
