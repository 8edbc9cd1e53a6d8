// merge_append.cu -- the two small kernels of the hot path:
//   * merge:  log-sum-exp merge of the pieces of units that straddled CTAs
//             (softmax over a union of disjoint key sets: lse = log sum_s e^lse_s,
//              out = sum_s e^(lse_s - lse) out_s);
//   * append: RoPE on the drafter's new q and k, then the store of k / v into
//             the draft slots (App. B: draft positions j > t take the drafter's
//             own K/V; Sec. 3.2: RoPE re-applied to drafted keys).
#include "kvshot_attn_common.cuh"

namespace kvshot {
namespace {

using namespace dev;

constexpr int kMergeThreads = 256;
constexpr int kMergeRows = kMergeThreads / 32;  // rows per CTA, one warp per row

// Workspace slot of the piece computed by CTA b is u + b.  One warp per row
// of a unit.  Launched behind the attention kernel with programmatic stream
// serialization, so its CTAs start as the attention CTAs leave.  Each warp
// first rebuilds the attention kernel's plan from the inputs alone (lengths ->
// tiles per unit -> the unit's tile range -> the CTAs that held it): rows of
// units that lived in one CTA leave at once, and the others only then wait
// for the attention grid, with one round of loads left: every piece's lse
// (lane k: piece b0 + k) together with the first two pieces' outputs (lane: 4
// dims).
// 6 resident CTAs per SM (<= 40 registers): a unit's rows for every split unit of the largest
// per-level plans fit in one wave, so no merge CTA waits for another to finish.
__global__ void __launch_bounds__(kMergeThreads, 6) merge_kernel(const __grid_constant__ AttnParams p) {
  const int blocks_per_unit = (p.rows_per_unit + kMergeRows - 1) / kMergeRows;
  const int u = blockIdx.x / blocks_per_unit;
  const int r = (blockIdx.x - u * blocks_per_unit) * kMergeRows + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int HR = p.hkv * p.row_blocks;
  const int c = u / HR, hr = u - c * HR;
  const int h = hr / p.row_blocks, rb = hr - h * p.row_blocks;
  const int rr = rb * p.rows_per_unit + r;
  if (r >= p.rows_per_unit || rr >= p.rows_total) return;
  // First tile of cache c and the total (the prefix sums of build_plan), 32 caches per round.
  int cbase = 0, total = 0, ut = 0;
  for (int c0 = 0; c0 < p.C; c0 += 32) {
    const int cc = c0 + lane;
    const int utc = cc < p.C ? (clamp_len(p, cc) + kTileKeys - 1) / kTileKeys + p.draft_tiles : 0;
    int below = cc < c ? utc * HR : 0, all = utc * HR;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      below += __shfl_xor_sync(0xffffffffu, below, o);
      all += __shfl_xor_sync(0xffffffffu, all, o);
    }
    cbase += below;
    total += all;
    if (c - c0 >= 0 && c - c0 < 32) ut = __shfl_sync(0xffffffffu, utc, c - c0);
  }
  const int gs = cbase + hr * ut;
  const int tpc = tiles_per_cta(total, p.num_ctas);
  const int b0 = gs / tpc, b1 = (gs + ut - 1) / tpc;
  if (b0 == b1) return;  // the unit lived in one CTA, which wrote the output itself
  wait_for_prerequisite_grid();
  const int np = b1 - b0 + 1;
  const int nl = rr / p.G, g = rr - nl * p.G;
  const size_t orow = (static_cast<size_t>(c) * p.Nq + nl) * p.hq + h * p.G + g;
  const size_t row0 = static_cast<size_t>(u + b0) * p.rows_per_unit + r;  // piece k's row: row0 + k * rows
  float ls = lane < np ? p.ws_lse[row0 + static_cast<size_t>(lane) * p.rows_per_unit] : -INFINITY;
  const int ostride = p.rows_per_unit * (kHeadDim / 4);  // float4s from one piece's row to the next's
  const float4* op = reinterpret_cast<const float4*>(p.ws_o + row0 * kHeadDim) + lane;
  const float4 v0 = op[0];  // np >= 2 here
  const float4 v1 = op[ostride];
  op += 2 * ostride;  // piece 2
  float M = ls;
  for (int k = lane + 32; k < np; k += 32)  // more than 32 pieces: fold the rest into this lane's max
    M = fmaxf(M, p.ws_lse[row0 + static_cast<size_t>(k) * p.rows_per_unit]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float Lsum = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (M != -INFINITY) {
    for (int k0 = 0; k0 < np; k0 += 32) {
      float wl = 0.f;
      if (k0 + lane < np) {
        const float lk = k0 == 0 ? ls : p.ws_lse[row0 + static_cast<size_t>(k0 + lane) * p.rows_per_unit];
        wl = lk == -INFINITY ? 0.f : exp2f(lk - M);
      }
      const int n = min(32, np - k0);
      for (int j = 0; j < n; ++j) {
        const float w = __shfl_sync(0xffffffffu, wl, j);
        Lsum += w;
        const int k = k0 + j;
        float4 x = v0;
        if (k == 1) {
          x = v1;
        } else if (k > 1) {
          x = *op;
          op += ostride;
        }
        acc.x += w * x.x;
        acc.y += w * x.y;
        acc.z += w * x.z;
        acc.w += w * x.w;
      }
    }
  }
  const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
  uint2 packed;
  packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2*>(p.out + orow * kHeadDim + 4 * lane) = packed;
  if (lane == 0) p.lse[orow] = Lsum > 0.f ? (M + log2f(Lsum)) * 0.69314718055994531f : -INFINITY;
}

constexpr int kAppendThreads = 256;

// One rotated component of RoPE, x' = a * cos - b * sin (sgn = -1) or
// y' = b * cos + a * sin (sgn = +1), rounded to bf16 as the fp64 evaluation
// rounds.  The fp32 value r differs from the exact a c + sgn b s by at most
// 2^-24 (|a| + 2 |b| + |r|) (cos/sin rounded to fp32, one product and one fma
// rounded); when r lies farther than twice that from every bf16 rounding
// midpoint both round alike, otherwise the component is recomputed in fp64.
__device__ __forceinline__ __nv_bfloat16 rope_bf16(float a, float b, float c32, float s32, double c, double s,
                                                   float sgn) {
  const float r = fmaf(a, c32, sgn * (b * s32));
  const uint32_t u = __float_as_uint(r);
  const int e = static_cast<int>((u >> 23) & 0xFFu);
  const float bound = 0x1p-23f * (fabsf(a) + 2.f * fabsf(b) + fabsf(r));
  if (e >= 40) {
    const float ulp = __uint_as_float(static_cast<uint32_t>(e - 23) << 23);  // 2^(e - 150), fp32 spacing at r
    const float dist = fabsf(static_cast<float>(static_cast<int>(u & 0xFFFFu) - 0x8000)) * ulp;
    if (dist > bound) return __float2bfloat16_rn(r);
  }
  const double da = a, db = b;
  return __double2bfloat16(sgn < 0.f ? da * c - db * s : da * c + db * s);
}

// One CTA per (cache, new node).  Work item = (head, 16-byte chunk j0 of the
// first half): it rotates dims j0..j0+7 together with their partners +64.
__global__ void __launch_bounds__(kAppendThreads) append_kernel(const __grid_constant__ AppendParams a) {
  // An attention call launched with KVSHOT_OVERLAP_PREVIOUS may start its prologue meanwhile.
  if (threadIdx.x == 0) allow_dependent_launch();
  __shared__ double s_cos[kHeadDim / 2], s_sin[kHeadDim / 2];
  const int c = blockIdx.x / a.n_new, i = blockIdx.x - (blockIdx.x / a.n_new) * a.n_new;
  const int pos = a.positions[static_cast<size_t>(c) * a.n_new + i];
  for (int j = threadIdx.x; j < kHeadDim / 2; j += blockDim.x) {
    double sn, cs;
    sincos(static_cast<double>(pos) * a.inv_freq[j], &sn, &cs);
    s_cos[j] = cs;
    s_sin[j] = sn;
  }
  __syncthreads();
  const int heads = a.hq + a.hkv;
  for (int w = threadIdx.x; w < heads * 8; w += blockDim.x) {
    const int head = w >> 3, j0 = (w & 7) * 8;
    const __nv_bfloat16* src;
    __nv_bfloat16* dst;
    if (head < a.hq) {
      const size_t off = ((static_cast<size_t>(c) * a.n_new + i) * a.hq + head) * kHeadDim;
      src = a.q_in + off;
      dst = a.q_out + off;
    } else {
      const int kh = head - a.hq;
      src = a.k_in + ((static_cast<size_t>(c) * a.n_new + i) * a.hkv + kh) * kHeadDim;
      dst = a.draft_k + ((static_cast<size_t>(c) * a.hkv + kh) * a.n_max + a.n0 + i) * kHeadDim;
    }
    const uint4 lo = *reinterpret_cast<const uint4*>(src + j0);
    const uint4 hi = *reinterpret_cast<const uint4*>(src + 64 + j0);
    const uint32_t wl[4] = {lo.x, lo.y, lo.z, lo.w}, wh[4] = {hi.x, hi.y, hi.z, hi.w};
    uint32_t ol[4], oh[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      __nv_bfloat16 rl[2], rh[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = j0 + 2 * k + e;
        const float x = e ? bf16_hi(wl[k]) : bf16_lo(wl[k]);
        const float y = e ? bf16_hi(wh[k]) : bf16_lo(wh[k]);
        const double cs = s_cos[j], sn = s_sin[j];
        const float c32 = static_cast<float>(cs), s32 = static_cast<float>(sn);
        rl[e] = rope_bf16(x, y, c32, s32, cs, sn, -1.f);
        rh[e] = rope_bf16(y, x, c32, s32, cs, sn, 1.f);
      }
      ol[k] = static_cast<uint32_t>(__bfloat16_as_ushort(rl[0])) |
              (static_cast<uint32_t>(__bfloat16_as_ushort(rl[1])) << 16);
      oh[k] = static_cast<uint32_t>(__bfloat16_as_ushort(rh[0])) |
              (static_cast<uint32_t>(__bfloat16_as_ushort(rh[1])) << 16);
    }
    *reinterpret_cast<uint4*>(dst + j0) = make_uint4(ol[0], ol[1], ol[2], ol[3]);
    *reinterpret_cast<uint4*>(dst + 64 + j0) = make_uint4(oh[0], oh[1], oh[2], oh[3]);
  }
  // V: plain copy into the draft slot.
  for (int w = threadIdx.x; w < a.hkv * 16; w += blockDim.x) {
    const int kh = w >> 4, ch = w & 15;
    const uint4 v = *reinterpret_cast<const uint4*>(
        a.v_in + ((static_cast<size_t>(c) * a.n_new + i) * a.hkv + kh) * kHeadDim + ch * 8);
    *reinterpret_cast<uint4*>(a.draft_v + ((static_cast<size_t>(c) * a.hkv + kh) * a.n_max + a.n0 + i) * kHeadDim +
                              ch * 8) = v;
  }
}

// QK-norm variant (Qwen3's per-head RMSNorm of q and k before RoPE): one warp per head, lane l
// holding dims 2l, 2l + 1 and their RoPE partners + 64.  x <- x / sqrt(mean(x^2) + eps) * w (w the
// head-dim weights), then the rotation; fp32 throughout, one rounding to bf16.
__global__ void __launch_bounds__(kAppendThreads) append_qknorm_kernel(const __grid_constant__ AppendParams a) {
  if (threadIdx.x == 0) allow_dependent_launch();
  __shared__ float s_cos[kHeadDim / 2], s_sin[kHeadDim / 2];
  const int c = blockIdx.x / a.n_new, i = blockIdx.x - (blockIdx.x / a.n_new) * a.n_new;
  const int pos = a.positions[static_cast<size_t>(c) * a.n_new + i];
  for (int j = threadIdx.x; j < kHeadDim / 2; j += blockDim.x) {
    double sn, cs;
    sincos(static_cast<double>(pos) * a.inv_freq[j], &sn, &cs);
    s_cos[j] = static_cast<float>(cs);
    s_sin[j] = static_cast<float>(sn);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = 2 * lane;
  for (int head = warp; head < a.hq + a.hkv; head += kAppendThreads / 32) {
    const __nv_bfloat16* src;
    __nv_bfloat16* dst;
    const __nv_bfloat16* w;
    if (head < a.hq) {
      const size_t off = ((static_cast<size_t>(c) * a.n_new + i) * a.hq + head) * kHeadDim;
      src = a.q_in + off;
      dst = a.q_out + off;
      w = a.q_norm_w;
    } else {
      const int kh = head - a.hq;
      src = a.k_in + ((static_cast<size_t>(c) * a.n_new + i) * a.hkv + kh) * kHeadDim;
      dst = a.draft_k + ((static_cast<size_t>(c) * a.hkv + kh) * a.n_max + a.n0 + i) * kHeadDim;
      w = a.k_norm_w;
    }
    const uint32_t lo = *reinterpret_cast<const uint32_t*>(src + j);
    const uint32_t hi = *reinterpret_cast<const uint32_t*>(src + 64 + j);
    const uint32_t wl = *reinterpret_cast<const uint32_t*>(w + j);
    const uint32_t wh = *reinterpret_cast<const uint32_t*>(w + 64 + j);
    float x[4] = {bf16_lo(lo), bf16_hi(lo), bf16_lo(hi), bf16_hi(hi)};
    float ss = x[0] * x[0] + x[1] * x[1] + x[2] * x[2] + x[3] * x[3];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float r = rsqrtf(ss * (1.f / kHeadDim) + a.eps);
    x[0] *= r * bf16_lo(wl);
    x[1] *= r * bf16_hi(wl);
    x[2] *= r * bf16_lo(wh);
    x[3] *= r * bf16_hi(wh);
    const float c0 = s_cos[j], s0 = s_sin[j], c1 = s_cos[j + 1], s1 = s_sin[j + 1];
    const float y0 = x[0] * c0 - x[2] * s0, y1 = x[1] * c1 - x[3] * s1;   // dims j, j + 1
    const float z0 = x[2] * c0 + x[0] * s0, z1 = x[3] * c1 + x[1] * s1;   // dims j + 64, j + 65
    *reinterpret_cast<uint32_t*>(dst + j) = pack_bf16x2(y0, y1);
    *reinterpret_cast<uint32_t*>(dst + 64 + j) = pack_bf16x2(z0, z1);
  }
  for (int w = threadIdx.x; w < a.hkv * 16; w += blockDim.x) {  // V: plain copy into the draft slot
    const int kh = w >> 4, ch = w & 15;
    const uint4 v = *reinterpret_cast<const uint4*>(
        a.v_in + ((static_cast<size_t>(c) * a.n_new + i) * a.hkv + kh) * kHeadDim + ch * 8);
    *reinterpret_cast<uint4*>(a.draft_v + ((static_cast<size_t>(c) * a.hkv + kh) * a.n_max + a.n0 + i) * kHeadDim +
                              ch * 8) = v;
  }
}

}  // namespace

cudaError_t launch_merge(const AttnParams& p, cudaStream_t stream) {
  const int units = p.C * p.hkv * p.row_blocks;
  const int blocks = units * ((p.rows_per_unit + kMergeRows - 1) / kMergeRows);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks);
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_kernel, p);
}

cudaError_t launch_append(const AppendParams& a, cudaStream_t stream) {
  if (a.q_norm_w != nullptr)
    append_qknorm_kernel<<<a.C * a.n_new, kAppendThreads, 0, stream>>>(a);
  else
    append_kernel<<<a.C * a.n_new, kAppendThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace kvshot
