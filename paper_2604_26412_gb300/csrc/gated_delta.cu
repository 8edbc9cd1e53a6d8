// gated_delta.cu -- the hybrid drafter's gated-delta fusion (Sec. 3.4,
// Eqs. "delta" and "fusion"): for every draft token, with n the
// self-attention branch (EAGLE-3 path) and o the cross-attention branch
// (re-attention to the target KV, the draft-attention call of this library),
//
//   delta = o - n
//   g     = sigmoid(W_g [n; o; delta] + b_g)      W_g in R^{d x 3d}, b_g in R^d
//   h     = n + g (.) (W_delta delta)             W_delta in R^{d x d}
//
// Two kernels.  The slab GEMM (kvshot_slab_gemm.cuh, tcgen05 tensor cores)
// computes the four products of the weight blocks with the token activations,
// one table entry each:
//   0: W_g[:, 0:d]   n          2: W_g[:, 2d:3d] o - W_g[:, 2d:3d] n
//   1: W_g[:, d:2d]  o          3: W_delta o - W_delta n
// delta is never rounded to bf16: entries 2 and 3 either multiply their
// weights by n and o stacked along the token axis and subtract the two fp32
// products (up to 128 tokens per block), or accumulate W o and the
// negated-weight product W n into one fp32 accumulator (larger blocks); both
// equal the product with the exact delta up to fp32 rounding.  Each
// product lands in a workspace slab [4][T][d].  gated_delta_finish, launched
// behind it with programmatic stream serialization, adds the slabs and
// applies the gate: h = n + sigmoid(slab0 + slab1 + slab2 + b_g) * slab3,
// rounded to bf16.
//
// The step is bound by the weights' bytes (4 d^2 bf16 values, read once:
// each weight tile is read by the CTAs of every token block at the same time,
// since the token block is the grid's fastest index) for the token counts of
// per-depth drafting; at a few hundred tokens it reaches the tensor pipe.
#include <algorithm>

#include "kvshot_slab_gemm.cuh"

namespace kvshot {
namespace {

using namespace dev;

constexpr int kFinishThreads = 256;
constexpr int kMaxFusionHidden = 32768;

struct FusionParams {
  const __nv_bfloat16* n;
  const __nv_bfloat16* b_g;
  __nv_bfloat16* h;
  const float* slab;  // [4][T][d]
  int T, d;
};

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
  if (d->hidden % sg::kFeat != 0 || d->hidden > kMaxFusionHidden) return KVSHOT_ERR_UNSUPPORTED;
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
  sg::Params gp;
  gp.slab = static_cast<float*>(d->workspace);
  gp.err = d->err_flag;
  gp.T = T;
  gp.d_out = D;
  gp.box_tok = std::min(T, sg::kMaxTok);
  const int nk = D / sg::kKT;
  // weight maps: 0 = W_g, 1 = W_delta; activation maps: 0 = n, 1 = o
  gp.e[0] = sg::Entry{0, 0, -1, 0, 0, 0, nk};      // W_g[:, 0:d] n
  gp.e[1] = sg::Entry{0, 1, -1, 0, D, 0, nk};      // W_g[:, d:2d] o
  gp.e[2] = sg::Entry{0, 0, 1, 0, 2 * D, 0, nk};   // W_g[:, 2d:3d] (o - n)
  gp.e[3] = sg::Entry{1, 0, 1, 0, 0, 0, nk};       // W_delta (o - n)
  sg::Maps maps;
  if (!encode_bf16_2d(&maps.w[0], w_g, 3 * static_cast<uint64_t>(D), D, sg::kKT, sg::kFeat) ||
      !encode_bf16_2d(&maps.w[1], w_delta, D, D, sg::kKT, sg::kFeat) ||
      !encode_bf16_2d(&maps.a[0], n, D, T, sg::kKT, static_cast<uint32_t>(gp.box_tok)) ||
      !encode_bf16_2d(&maps.a[1], o, D, T, sg::kKT, static_cast<uint32_t>(gp.box_tok)))
    return KVSHOT_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (sg::launch(gp, maps, 4, s) != cudaSuccess) return KVSHOT_ERR_CUDA;
  FusionParams p;
  p.n = static_cast<const __nv_bfloat16*>(n);
  p.b_g = static_cast<const __nv_bfloat16*>(b_g);
  p.h = static_cast<__nv_bfloat16*>(h);
  p.slab = gp.slab;
  p.T = T;
  p.d = D;
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
  return cudaLaunchKernelEx(&cfg, gated_delta_finish, p) == cudaSuccess ? KVSHOT_OK : KVSHOT_ERR_CUDA;
}
