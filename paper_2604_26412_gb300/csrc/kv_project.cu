// kv_project.cu -- the KV-only drafter's linear projection of multi-layer
// target KV (Sec. 3.2, injection strategy "linear projection", with the
// "Proj + RoPE fix" variant): for every newly verified token t the K (and V)
// vectors of the L_s sampled target layers, each hkv x 128 wide, are
// concatenated and mapped back to one layer's width by learned matrices
// W_K^proj, W_V^proj in R^{d_kv x L_s d_kv} (d_kv = hkv x 128):
//
//   K'(t) = W_K^proj [K^(1)(t); ...; K^(L_s)(t)],   V'(t) = W_V^proj [V^(1)(t); ...; V^(L_s)(t)]
//
// and, with KVSHOT_PROJECT_ROPE, RoPE is re-applied to K'(t) at the token's
// position (the projection mixes keys already rotated by RoPE).  The results
// go to the token's slot of the single reused cache the draft attention reads
// (App. B: verified prefix positions take the target's -- here projected --
// K/V), so the cache is built incrementally, a few tokens per decoding step.
//
// Two kernels.  The slab GEMM (kvshot_slab_gemm.cuh) computes the products per
// layer block (table entry (K or V, layer l): W[:, l d_kv : (l+1) d_kv] times
// the tokens' layer-l K or V), into fp32 slabs [2 L_s][T][d_kv].
// kv_project_finish adds each output's L_s slabs, rotates the keys, rounds to
// bf16 and stores both vectors into the cache through the page table.  The
// angle pos * rope_base^(-2j/128) is formed and reduced modulo 2 pi in fp64
// (from a host table of the frequencies); sine, cosine and the rotation are
// fp32 (relative error ~1e-7, far below the bf16 rounding that follows).
// fp64 sine and cosine cost this latency-bound kernel ~2 us per call on GB300.
#include <algorithm>
#include <cmath>

#include "kvshot_slab_gemm.cuh"

namespace kvshot {
namespace {

using namespace dev;

constexpr int kFinishThreads = 256;  // (token, KV head) pairs of 64 rotation pairs: 4 per CTA
constexpr int kMaxLayers = sg::kMaxEntries / 2;

struct ProjectParams {
  const float* slab;  // [2 L][T][d_kv]
  const int32_t* token_cache;
  const int32_t* positions;
  const int32_t* page_table;  // null: contiguous cache
  __nv_bfloat16* k_out;
  __nv_bfloat16* v_out;
  int32_t* err;
  int T, L, hkv, C;
  int paged, page_size, max_pages, num_pages, l_cap;
  int rope;
  double inv_freq[kHeadDim / 2];  // rope_base^(-2j/128), fp64
};

// One thread per (token, KV head, rotation pair j in [0, 64)): features j and j + 64 of the head.
__global__ void __launch_bounds__(kFinishThreads) kv_project_finish(const __grid_constant__ ProjectParams p) {
  wait_for_prerequisite_grid();
  const int dkv = p.hkv * kHeadDim;
  const int g = blockIdx.x * (kFinishThreads / 64) + (threadIdx.x >> 6);  // (token, head)
  const int j = threadIdx.x & 63;
  if (g >= p.T * p.hkv) return;
  const int t = g / p.hkv, h = g - t * p.hkv;
  const int c = p.token_cache[t], pos = p.positions[t];
  const int cap = p.paged ? p.max_pages * p.page_size : p.l_cap;
  if (c < 0 || c >= p.C || pos < 0 || pos >= cap) {
    if (j == 0) set_error(p.err, KVSHOT_ERR_DEVICE_BOUNDS);
    return;
  }
  size_t row;
  if (p.paged) {
    const int pid = p.page_table[static_cast<size_t>(c) * p.max_pages + pos / p.page_size];
    if (pid < 0 || pid >= p.num_pages) {
      if (j == 0) set_error(p.err, KVSHOT_ERR_DEVICE_BOUNDS);
      return;
    }
    row = (static_cast<size_t>(pid) * p.hkv + h) * p.page_size + pos % p.page_size;
  } else {
    row = (static_cast<size_t>(c) * p.hkv + h) * p.l_cap + pos;
  }
  const size_t td = static_cast<size_t>(p.T) * dkv;
  const size_t f = static_cast<size_t>(t) * dkv + h * kHeadDim + j;
  float kx = 0.f, ky = 0.f, vx = 0.f, vy = 0.f;
  for (int l = 0; l < p.L; ++l) {
    kx += p.slab[l * td + f];
    ky += p.slab[l * td + f + 64];
    vx += p.slab[(p.L + l) * td + f];
    vy += p.slab[(p.L + l) * td + f + 64];
  }
  if (p.rope) {
    const double a = static_cast<double>(pos) * p.inv_freq[j];
    const double r = a - 6.283185307179586 * rint(a * 0.15915494309189535);
    float sn, cs;
    sincosf(static_cast<float>(r), &sn, &cs);
    const float x = kx, y = ky;
    kx = x * cs - y * sn;
    ky = y * cs + x * sn;
  }
  p.k_out[row * kHeadDim + j] = __float2bfloat16_rn(kx);
  p.k_out[row * kHeadDim + j + 64] = __float2bfloat16_rn(ky);
  p.v_out[row * kHeadDim + j] = __float2bfloat16_rn(vx);
  p.v_out[row * kHeadDim + j + 64] = __float2bfloat16_rn(vy);
}

bool aligned(const void* ptr, size_t a) { return (reinterpret_cast<uintptr_t>(ptr) % a) == 0; }

size_t slab_bytes(const kvshot_project_desc* d) {
  return static_cast<size_t>(2) * d->num_layers * static_cast<size_t>(d->num_tokens) * d->hkv * kHeadDim * 4;
}

kvshot_status check_desc(const kvshot_project_desc* d, bool paged) {
  if (d == nullptr) return KVSHOT_ERR_NULL;
  if (d->num_tokens < 0 || d->num_layers < 1 || d->hkv < 1 || d->num_caches < 1) return KVSHOT_ERR_SHAPE;
  if (d->head_dim != kHeadDim || d->num_layers > kMaxLayers || d->hkv > 64) return KVSHOT_ERR_UNSUPPORTED;
  if (!(d->rope_base > 0.f) || !std::isfinite(d->rope_base)) return KVSHOT_ERR_SHAPE;
  if ((d->flags & ~KVSHOT_PROJECT_ROPE) != 0) return KVSHOT_ERR_SHAPE;
  if (static_cast<int64_t>(d->num_tokens) * d->num_layers * d->hkv * kHeadDim >= (int64_t(1) << 31))
    return KVSHOT_ERR_UNSUPPORTED;
  if (paged) {
    if (d->page_size < 1 || d->max_pages_per_seq < 1 || d->num_pages < 1) return KVSHOT_ERR_SHAPE;
  } else if (d->l_cap < 1) {
    return KVSHOT_ERR_SHAPE;
  }
  return KVSHOT_OK;
}

}  // namespace
}  // namespace kvshot

using namespace kvshot;

extern "C" size_t kvshot_kv_project_workspace_size(const kvshot_project_desc* d) {
  if (d == nullptr || check_desc(d, d->page_size > 0) != KVSHOT_OK) return 0;
  return std::max<size_t>(256, slab_bytes(d));
}

extern "C" kvshot_status kvshot_kv_project(const kvshot_project_desc* d, const void* k_in, const void* v_in,
                                           const void* w_k, const void* w_v, const int32_t* token_cache,
                                           const int32_t* positions, const int32_t* page_table, void* k_out,
                                           void* v_out, kvshot_stream_t stream) {
  const bool paged = page_table != nullptr;
  if (kvshot_status st = check_desc(d, paged)) return st;
  if (d->num_tokens == 0) return KVSHOT_OK;
  if (!k_in || !v_in || !w_k || !w_v || !token_cache || !positions || !k_out || !v_out) return KVSHOT_ERR_NULL;
  if (!aligned(k_in, 16) || !aligned(v_in, 16) || !aligned(w_k, 16) || !aligned(w_v, 16) || !aligned(k_out, 16) ||
      !aligned(v_out, 16) || !aligned(token_cache, 4) || !aligned(positions, 4) || (paged && !aligned(page_table, 4)))
    return KVSHOT_ERR_ALIGN;
  if (d->workspace == nullptr || !aligned(d->workspace, 256) || d->workspace_bytes < slab_bytes(d))
    return KVSHOT_ERR_WORKSPACE;
  const int T = d->num_tokens, L = d->num_layers, dkv = d->hkv * kHeadDim;
  sg::Params gp;
  gp.slab = static_cast<float*>(d->workspace);
  gp.err = d->err_flag;
  gp.T = T;
  gp.d_out = dkv;
  gp.box_tok = std::min(T, sg::kMaxTok);
  // weight maps: 0 = W_K, 1 = W_V; activation maps: 0 = K of the L layers, 1 = V ([T, L d_kv] rows)
  for (int l = 0; l < L; ++l) {
    gp.e[l] = sg::Entry{0, 0, -1, 0, l * dkv, l * dkv, dkv / sg::kKT};
    gp.e[L + l] = sg::Entry{1, 1, -1, 0, l * dkv, l * dkv, dkv / sg::kKT};
  }
  const uint64_t K = static_cast<uint64_t>(L) * dkv;
  sg::Maps maps;
  if (!encode_bf16_2d(&maps.w[0], w_k, K, dkv, sg::kKT, sg::kFeat) ||
      !encode_bf16_2d(&maps.w[1], w_v, K, dkv, sg::kKT, sg::kFeat) ||
      !encode_bf16_2d(&maps.a[0], k_in, K, T, sg::kKT, static_cast<uint32_t>(gp.box_tok)) ||
      !encode_bf16_2d(&maps.a[1], v_in, K, T, sg::kKT, static_cast<uint32_t>(gp.box_tok)))
    return KVSHOT_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (sg::launch(gp, maps, 2 * L, s) != cudaSuccess) return KVSHOT_ERR_CUDA;
  ProjectParams p;
  p.slab = gp.slab;
  p.token_cache = token_cache;
  p.positions = positions;
  p.page_table = page_table;
  p.k_out = static_cast<__nv_bfloat16*>(k_out);
  p.v_out = static_cast<__nv_bfloat16*>(v_out);
  p.err = d->err_flag;
  p.T = T;
  p.L = L;
  p.hkv = d->hkv;
  p.C = d->num_caches;
  p.paged = paged ? 1 : 0;
  p.page_size = paged ? d->page_size : 0;
  p.max_pages = paged ? d->max_pages_per_seq : 0;
  p.num_pages = paged ? d->num_pages : 0;
  p.l_cap = paged ? 0 : d->l_cap;
  p.rope = (d->flags & KVSHOT_PROJECT_ROPE) ? 1 : 0;
  for (int j = 0; j < kHeadDim / 2; ++j)
    p.inv_freq[j] = std::pow(static_cast<double>(d->rope_base), -2.0 * j / kHeadDim);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  const int pairs = T * d->hkv;  // (token, head) pairs, 4 per CTA
  cfg.gridDim = dim3(static_cast<unsigned>((pairs + kFinishThreads / 64 - 1) / (kFinishThreads / 64)));
  cfg.blockDim = dim3(kFinishThreads);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kv_project_finish, p) == cudaSuccess ? KVSHOT_OK : KVSHOT_ERR_CUDA;
}
