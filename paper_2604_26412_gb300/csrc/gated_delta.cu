// gated_delta.cu -- the hybrid drafter's gated-delta fusion (Sec. 3.4,
// Eqs. "delta" and "fusion"): for every draft token, with n the
// self-attention branch (EAGLE-3 path) and o the cross-attention branch
// (re-attention to the target KV, the draft-attention call of this library),
//
//   delta = o - n
//   g     = sigmoid(W_g [n; o; delta] + b_g)      W_g in R^{d x 3d}, b_g in R^d
//   h     = n + g (.) (W_delta delta)             W_delta in R^{d x d}
//
// Two kernels.  gated_delta_gemm computes the four products of the weight
// blocks with the token activations on the tcgen05 tensor cores (A = a
// 128-row block of weights, K-major; B = a block of up to 128 tokens,
// K-major; fp32 accumulators in TMEM), one weight block per CTA row of the
// grid:
//   block 0: W_g[:, 0:d]   n          block 2: W_g[:, 2d:3d] o - W_g[:, 2d:3d] n
//   block 1: W_g[:, d:2d]  o          block 3: W_delta o - W_delta n
// delta is never rounded to bf16: blocks 2 and 3 multiply their weights by
// n and o stacked along the token axis (one MMA of N = 256) and subtract the
// two fp32 products, which equals the product with the exact delta up to fp32
// rounding.  Each CTA writes its fp32 result for its (feature block, token
// block) to a workspace slab [4][T][d].  gated_delta_finish, launched behind it
// with programmatic stream serialization, adds the slabs and applies the gate:
// h = n + sigmoid(slab0 + slab1 + slab2 + b_g) * slab3, rounded to bf16.
//
// The step is bound by the weights' bytes (4 d^2 bf16 values, read once:
// each weight tile is read by the CTAs of every token block at the same time,
// since the token block is the grid's fastest index) for the token counts of
// per-depth drafting; at a few hundred tokens it reaches the tensor pipe.
#include <algorithm>

#include "kvshot_attn_common.cuh"
#include "kvshot_tcgen05.cuh"

namespace kvshot {
namespace {

using namespace dev;
using namespace tc;

constexpr int kFeat = 128;                    // output features per CTA (MMA M)
constexpr int kTok = 128;                     // tokens per CTA (MMA N per operand)
constexpr int kKT = 64;                       // K per stage: one 128-byte swizzled row
constexpr int kGemmStages = 6;                // ring slots: blocks 0/1 use all 6 (32 KB each), blocks 2/3 four (48 KB)
constexpr int kGemmThreads = 128;             // warp 0 lane 0: TMA; warp 1: TMEM owner, lane 0 MMA; all: epilogue
constexpr int kABytes = kFeat * kKT * 2;      // 16 KB
constexpr int kBBytes = 2 * kTok * kKT * 2;   // 32 KB: n rows then o rows
constexpr uint32_t kGemmTmemCols = 256;       // [0, 128): W n (or W o); [128, 256): W o
constexpr int kFinishThreads = 256;
constexpr int kMaxFusionHidden = 32768;

// 2-D tiled TMA load with the default L2 policy (activations: every feature block reads them).
__device__ __forceinline__ void tma_load_2d_nohint(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

struct FusionParams {
  const __nv_bfloat16* n;
  const __nv_bfloat16* b_g;
  __nv_bfloat16* h;
  float* slab;   // [4][T][d]
  int32_t* err;
  int T, d;
  int box_tok;   // token rows per TMA box of n / o: min(T, 128)
};

struct FusionMaps {
  CUtensorMap wg;  // W_g [d, 3d], boxes {64, 128}
  CUtensorMap wd;  // W_delta [d, d], boxes {64, 128}
  CUtensorMap n;   // n [T, d], boxes {64, box_tok}
  CUtensorMap o;   // o [T, d], boxes {64, box_tok}
};

constexpr int kRingBytes = 4 * (kABytes + kBBytes);  // 192 KB: 6 x (A + one token tile) or 4 x (A + two)

size_t gemm_smem_bytes() { return 1024 + kRingBytes + 8 * (2 * kGemmStages + 1) + 16; }

// Grid (token blocks, feature blocks, 4 weight blocks).
__global__ void __launch_bounds__(kGemmThreads, 1)
    gated_delta_gemm(const __grid_constant__ FusionParams p, const __grid_constant__ FusionMaps maps) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();
  const int tt = blockIdx.x, ft = blockIdx.y, blk = blockIdx.z;
  const bool both = blk >= 2;  // B holds the n rows and the o rows
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // Ring slot s: A at base + s * slot, B right after it (one or two token tiles).
  const int nst = both ? 4 : 6;
  const int slot = kABytes + (both ? 2 : 1) * kTok * 128;
  uint64_t* full = reinterpret_cast<uint64_t*>(base + kRingBytes);
  uint64_t* empty = full + kGemmStages;
  uint64_t* done = empty + kGemmStages;
  uint32_t* tmem_base = reinterpret_cast<uint32_t*>(done + 1);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), 1);
    }
    mbar_init(smem_addr(done), 1);
    fence_mbar_init();
    prefetch_tensormap(blk == 3 ? &maps.wd : &maps.wg);
    prefetch_tensormap(&maps.n);
    prefetch_tensormap(&maps.o);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_base), kGemmTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base;
  const int nk = p.d / kKT;
  bool ok = true;
  if (warp == 0 && lane == 0) {
    const uint64_t stream_once = l2_policy_evict_first();  // weights: read once
    const CUtensorMap* wmap = blk == 3 ? &maps.wd : &maps.wg;
    const int wx0 = blk == 3 ? 0 : blk * p.d;
    const uint32_t tx = kABytes + (both ? 2 : 1) * p.box_tok * 128;
    for (int kt = 0; kt < nk && ok; ++kt) {
      const int s = kt % nst;
      if (kt >= nst) ok = mbar_wait(smem_addr(&empty[s]), ((kt - nst) / nst) & 1, p.err);
      if (!ok) break;
      const uint32_t fb = smem_addr(&full[s]);
      mbar_arrive_expect_tx(fb, tx);
      tma_load_2d(smem_addr(base + s * slot), wmap, wx0 + kt * kKT, ft * kFeat, fb, stream_once);
      const uint32_t bdst = smem_addr(base + s * slot + kABytes);
      const int ty = tt * kTok;
      if (blk == 1) {
        tma_load_2d_nohint(bdst, &maps.o, kt * kKT, ty, fb);
      } else {
        tma_load_2d_nohint(bdst, &maps.n, kt * kKT, ty, fb);
        if (both) tma_load_2d_nohint(bdst + kTok * 128, &maps.o, kt * kKT, ty, fb);
      }
    }
  } else if (warp == 1 && lane == 0) {
    const uint32_t idesc = idesc_bf16(kFeat, both ? 2 * kTok : kTok, false);
    for (int kt = 0; kt < nk && ok; ++kt) {
      const int s = kt % nst;
      ok = mbar_wait(smem_addr(&full[s]), (kt / nst) & 1, p.err);
      if (!ok) break;
      tc_fence_after();
      const uint32_t a0 = smem_addr(base + s * slot), b0 = a0 + kABytes;
#pragma unroll
      for (int ks = 0; ks < kKT / 16; ++ks) {
        const uint64_t a = smem_desc_sw128(a0 + ks * 32, 16, 1024);
        const uint64_t b = smem_desc_sw128(b0 + ks * 32, 16, 1024);
        tc_mma(tmem, a, b, idesc, (kt | ks) ? 1u : 0u);
      }
      tc_commit(smem_addr(&empty[s]));
    }
    tc_commit(smem_addr(done));  // every MMA this thread issued has completed
  }
  __syncwarp();
  // Epilogue: thread = TMEM lane = output feature; 32 tokens per TMEM load.
  ok = mbar_wait(smem_addr(done), 0, p.err);
  tc_fence_after();
  const int f = ft * kFeat + warp * 32 + lane;
  const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  float* slab = p.slab + static_cast<size_t>(blk) * p.T * p.d;
#pragma unroll 1
  for (int c = 0; c < kTok / 32; ++c) {
    const int t0 = tt * kTok + c * 32;
    if (t0 >= p.T) break;
    uint32_t x[32], y[32];
    tmem_ld32(trow + c * 32, x);
    if (both) tmem_ld32(trow + kTok + c * 32, y);
    tmem_wait_ld();
    const int nt = min(32, p.T - t0);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float v = both ? __uint_as_float(y[j]) - __uint_as_float(x[j]) : __uint_as_float(x[j]);
      if (j < nt) slab[static_cast<size_t>(t0 + j) * p.d + f] = ok ? v : 0.f;  // a warp stores 32 consecutive features
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, kGemmTmemCols);
}

__device__ __forceinline__ float sigmoid(float z) { return 1.f / (1.f + __expf(-z)); }

// h = n + sigmoid(slab0 + slab1 + slab2 + b_g) * slab3, four features per thread.
__global__ void __launch_bounds__(kFinishThreads) gated_delta_finish(const __grid_constant__ FusionParams p) {
  wait_for_prerequisite_grid();
  const size_t td = static_cast<size_t>(p.T) * p.d;
  const size_t e = (static_cast<size_t>(blockIdx.x) * kFinishThreads + threadIdx.x) * 4;
  if (e >= td) return;
  const int f = static_cast<int>(e % p.d);
  const float4 s0 = *reinterpret_cast<const float4*>(p.slab + e);
  const float4 s1 = *reinterpret_cast<const float4*>(p.slab + td + e);
  const float4 s2 = *reinterpret_cast<const float4*>(p.slab + 2 * td + e);
  const float4 u = *reinterpret_cast<const float4*>(p.slab + 3 * td + e);
  const uint2 nb = *reinterpret_cast<const uint2*>(p.n + e);
  const uint2 bb = *reinterpret_cast<const uint2*>(p.b_g + f);
  const float2 n01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&nb.x));
  const float2 n23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&nb.y));
  const float2 b01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bb.x));
  const float2 b23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bb.y));
  const float h0 = n01.x + sigmoid(s0.x + s1.x + s2.x + b01.x) * u.x;
  const float h1 = n01.y + sigmoid(s0.y + s1.y + s2.y + b01.y) * u.y;
  const float h2 = n23.x + sigmoid(s0.z + s1.z + s2.z + b23.x) * u.z;
  const float h3 = n23.y + sigmoid(s0.w + s1.w + s2.w + b23.y) * u.w;
  uint2 out;
  out.x = pack_bf16x2(h0, h1);
  out.y = pack_bf16x2(h2, h3);
  *reinterpret_cast<uint2*>(p.h + e) = out;
}

bool aligned(const void* ptr, size_t a) { return (reinterpret_cast<uintptr_t>(ptr) % a) == 0; }

size_t slab_bytes(const kvshot_fusion_desc* d) {
  return static_cast<size_t>(4) * static_cast<size_t>(d->num_tokens) * static_cast<size_t>(d->hidden) * 4;
}

kvshot_status check_desc(const kvshot_fusion_desc* d) {
  if (d == nullptr) return KVSHOT_ERR_NULL;
  if (d->num_tokens < 0 || d->hidden <= 0) return KVSHOT_ERR_SHAPE;
  if (d->hidden % kFeat != 0 || d->hidden > kMaxFusionHidden) return KVSHOT_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(d->num_tokens) * d->hidden >= (int64_t(1) << 31)) return KVSHOT_ERR_UNSUPPORTED;
  return KVSHOT_OK;
}

}  // namespace
}  // namespace kvshot

using namespace kvshot;

extern "C" size_t kvshot_gated_delta_workspace_size(const kvshot_fusion_desc* d) {
  if (check_desc(d) != KVSHOT_OK) return 0;
  return std::max<size_t>(256, slab_bytes(d));
}

extern "C" kvshot_status kvshot_gated_delta(const kvshot_fusion_desc* d, const void* n, const void* o,
                                            const void* w_g, const void* b_g, const void* w_delta, void* h,
                                            kvshot_stream_t stream) {
  if (kvshot_status st = check_desc(d)) return st;
  if (d->num_tokens == 0) return KVSHOT_OK;
  if (!n || !o || !w_g || !b_g || !w_delta || !h) return KVSHOT_ERR_NULL;
  if (!aligned(n, 16) || !aligned(o, 16) || !aligned(w_g, 16) || !aligned(b_g, 8) || !aligned(w_delta, 16) ||
      !aligned(h, 8))
    return KVSHOT_ERR_ALIGN;
  if (d->workspace == nullptr || !aligned(d->workspace, 256) || d->workspace_bytes < slab_bytes(d))
    return KVSHOT_ERR_WORKSPACE;
  const int T = d->num_tokens, D = d->hidden;
  FusionParams p;
  p.n = static_cast<const __nv_bfloat16*>(n);
  p.b_g = static_cast<const __nv_bfloat16*>(b_g);
  p.h = static_cast<__nv_bfloat16*>(h);
  p.slab = static_cast<float*>(d->workspace);
  p.err = d->err_flag;
  p.T = T;
  p.d = D;
  p.box_tok = std::min(T, kTok);
  FusionMaps maps;
  if (!encode_bf16_2d(&maps.wg, w_g, 3 * static_cast<uint64_t>(D), D, kKT, kFeat) ||
      !encode_bf16_2d(&maps.wd, w_delta, D, D, kKT, kFeat) ||
      !encode_bf16_2d(&maps.n, n, D, T, kKT, static_cast<uint32_t>(p.box_tok)) ||
      !encode_bf16_2d(&maps.o, o, D, T, kKT, static_cast<uint32_t>(p.box_tok)))
    return KVSHOT_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t smem = gemm_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(gated_delta_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return KVSHOT_ERR_CUDA;
  const dim3 grid((T + kTok - 1) / kTok, D / kFeat, 4);
  gated_delta_gemm<<<grid, kGemmThreads, smem, s>>>(p, maps);
  if (cudaGetLastError() != cudaSuccess) return KVSHOT_ERR_CUDA;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  const size_t quads = static_cast<size_t>(T) * D / 4;
  cfg.gridDim = dim3(static_cast<unsigned>((quads + kFinishThreads - 1) / kFinishThreads));
  cfg.blockDim = dim3(kFinishThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, gated_delta_finish, p);
  return e == cudaSuccess ? KVSHOT_OK : KVSHOT_ERR_CUDA;
}
