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

constexpr int kMergeThreads = 128;

// One CTA per unit.  Workspace slot of the piece computed by CTA b is u + b.
__global__ void __launch_bounds__(kMergeThreads) merge_kernel(const __grid_constant__ AttnParams p) {
  const int u = blockIdx.x;
  const int HR = p.hkv * p.row_blocks;
  const int c = u / HR, hr = u - c * HR;
  const int h = hr / p.row_blocks, rb = hr - h * p.row_blocks;
  const int L = clamp_len(p, c);
  const int ut = (L + kTileKeys - 1) / kTileKeys + p.draft_tiles;
  const int gs = p.ws_meta[c] + hr * ut;
  const int total = p.ws_meta[p.C];
  const int tpc = tiles_per_cta(total, p.num_ctas);
  const int b0 = gs / tpc, b1 = (gs + ut - 1) / tpc;
  if (b0 == b1) return;  // the unit lived in one CTA, which wrote the output itself
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int r = warp; r < p.rows_per_unit; r += kMergeThreads / 32) {
    const int rr = rb * p.rows_per_unit + r;
    if (rr >= p.rows_total) break;
    float M = -INFINITY;
    for (int b = b0; b <= b1; ++b) M = fmaxf(M, p.ws_lse[static_cast<size_t>(u + b) * p.rows_per_unit + r]);
    float Lsum = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (M != -INFINITY) {
      for (int b = b0; b <= b1; ++b) {
        const size_t row = static_cast<size_t>(u + b) * p.rows_per_unit + r;
        const float ls = p.ws_lse[row];
        if (ls == -INFINITY) continue;
        const float w = exp2f(ls - M);
        Lsum += w;
        const float4 v = *reinterpret_cast<const float4*>(p.ws_o + row * kHeadDim + 4 * lane);
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
    }
    const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
    const int nl = rr / p.G, g = rr - nl * p.G;
    const size_t orow = (static_cast<size_t>(c) * p.Nq + nl) * p.hq + h * p.G + g;
    uint2 packed;
    packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
    packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(p.out + orow * kHeadDim + 4 * lane) = packed;
    if (lane == 0) p.lse[orow] = Lsum > 0.f ? (M + log2f(Lsum)) * 0.69314718055994531f : -INFINITY;
  }
}

constexpr int kAppendThreads = 256;

// One CTA per (cache, new node).  Work item = (head, 16-byte chunk j0 of the
// first half): it rotates dims j0..j0+7 together with their partners +64.
__global__ void __launch_bounds__(kAppendThreads) append_kernel(const __grid_constant__ AppendParams a) {
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
        const double x = e ? bf16_hi(wl[k]) : bf16_lo(wl[k]);
        const double y = e ? bf16_hi(wh[k]) : bf16_lo(wh[k]);
        rl[e] = __double2bfloat16(x * s_cos[j] - y * s_sin[j]);
        rh[e] = __double2bfloat16(y * s_cos[j] + x * s_sin[j]);
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

}  // namespace

cudaError_t launch_merge(const AttnParams& p, cudaStream_t stream) {
  const int units = p.C * p.hkv * p.row_blocks;
  merge_kernel<<<units, kMergeThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_append(const AppendParams& a, cudaStream_t stream) {
  append_kernel<<<a.C * a.n_new, kAppendThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace kvshot
