// attn_cc.cu -- draft attention for small GQA stacks (<= 4 query rows per KV
// head, e.g. one chain-drafting step with G = 4): CUDA-core dot products.
//
// At 4 rows the step does 4 flop per byte of K/V, well under the FMA ridge,
// so tensor cores would idle three quarters of each 16-row tile; the kernel
// instead spends its issue slots on fp32 FMAs over 16-byte shared-memory
// vectors.  Per tile each consumer warp owns 16 keys; a key is handled by 8
// lanes (16 dims each), its 4 row scores reduced with 3 xor-shuffles.
//
// Math: Sec. 2.2 Eq. "kv-reattention" (softmax re-attention of the drafter's
// query over reused target K/V) over the memory M_i of Sec. 3.4 / App. B,
// computed as an online softmax in the log2 domain; pieces of a unit split
// across CTAs are merged by the merge kernel (log-sum-exp of the pieces).
#include "kvshot_attn_common.cuh"

namespace kvshot {
namespace {

using namespace dev;

constexpr int kWarps = 4;                  // consumer warps
constexpr int kStages = 3;
constexpr int kThreads = (kWarps + 1) * 32;
constexpr int kKeysPerWarp = kTileKeys / kWarps;  // 16
constexpr int kIters = kKeysPerWarp / 4;          // 4 keys (4 lane groups) per iteration
constexpr int kBarConsumers = 1;

struct Smem {
  uint8_t* ring;
  uint64_t* full;
  uint64_t* empty;
  int* len;
  int* base;
  uint64_t* anc;
  int* par;
  float* comb_o;   // [kWarps][4][128]
  float* comb_m;   // [kWarps][4]
  float* comb_l;   // [kWarps][4]
  int* misc;       // [0] abort, [1] issued
};

__host__ __device__ inline size_t smem_bytes(int C) {
  size_t off = static_cast<size_t>(kStages) * kStageBytes;
  off += 2 * kStages * sizeof(uint64_t);
  off += sizeof(uint64_t) * kMaxTreeNodes;
  off += sizeof(int) * kMaxTreeNodes;
  off += sizeof(float) * kWarps * kCcRows * (kHeadDim + 2);
  off += sizeof(int) * 4;
  off += sizeof(int) * (2 * C + 1);
  return off + 1024;  // alignment slack for the ring
}

__device__ Smem carve(uint8_t* raw, int C) {
  Smem s;
  uint8_t* p = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  s.ring = p;
  p += kStages * kStageBytes;
  s.full = reinterpret_cast<uint64_t*>(p);
  s.empty = s.full + kStages;
  s.anc = s.empty + kStages;
  s.par = reinterpret_cast<int*>(s.anc + kMaxTreeNodes);
  s.comb_o = reinterpret_cast<float*>(s.par + kMaxTreeNodes);
  s.comb_m = s.comb_o + kWarps * kCcRows * kHeadDim;
  s.comb_l = s.comb_m + kWarps * kCcRows;
  s.misc = reinterpret_cast<int*>(s.comb_l + kWarps * kCcRows);
  s.len = s.misc + 4;
  s.base = s.len + C;
  return s;
}

__device__ __forceinline__ void unpack16(const uint4& a, const uint4& b, float (&f)[16]) {
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    f[2 * i] = bf16_lo(w[i]);
    f[2 * i + 1] = bf16_hi(w[i]);
  }
}

// Final or partial write of one unit piece: combine the 4 consumer warps'
// (m, l, o) states through shared memory.
__device__ __forceinline__ void finalize(const AttnParams& p, const Smem& sm, int c, int h, int rb, int slot, bool whole,
                         float (&o)[kCcRows][16], const float (&m_run)[kCcRows], float (&l_run)[kCcRows]) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane >> 3, s8 = lane & 7;
  // Sum the 4 lane groups (different keys, same running max).
#pragma unroll
  for (int r = 0; r < kCcRows; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 8);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 16);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      o[r][i] += __shfl_xor_sync(0xffffffffu, o[r][i], 8);
      o[r][i] += __shfl_xor_sync(0xffffffffu, o[r][i], 16);
    }
  }
  if (grp == 0) {
#pragma unroll
    for (int r = 0; r < kCcRows; ++r) {
      float* dst = sm.comb_o + (warp * kCcRows + r) * kHeadDim;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        dst[8 * s8 + i] = o[r][i];
        dst[64 + 8 * s8 + i] = o[r][8 + i];
      }
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int r = 0; r < kCcRows; ++r) {
      sm.comb_m[warp * kCcRows + r] = m_run[r];
      sm.comb_l[warp * kCcRows + r] = l_run[r];
    }
  }
  named_barrier_sync(kBarConsumers, kWarps * 32);
  // 128 threads: row = tid / 32, dims 4 * (tid % 32) .. +3.
  const int tid = threadIdx.x;
  const int r = tid >> 5, d0 = (tid & 31) * 4;
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm.comb_m[w * kCcRows + r]);
  float Lsum = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
  if (M != -INFINITY) {
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float mw = sm.comb_m[w * kCcRows + r];
      const float wt = mw == -INFINITY ? 0.f : ex2(mw - M);
      Lsum += wt * sm.comb_l[w * kCcRows + r];
      const float4 v = *reinterpret_cast<const float4*>(sm.comb_o + (w * kCcRows + r) * kHeadDim + d0);
      acc[0] += wt * v.x;
      acc[1] += wt * v.y;
      acc[2] += wt * v.z;
      acc[3] += wt * v.w;
    }
  }
  const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
  const float lse2 = Lsum > 0.f ? M + __log2f(Lsum) : -INFINITY;
  const int rr = rb * p.rows_per_unit + r;  // row within the unit's GQA stack
  if (r < p.rows_per_unit && rr < p.rows_total) {
    if (whole) {
      const int nl = rr / p.G, g = rr - nl * p.G;
      const size_t row = (static_cast<size_t>(c) * p.Nq + nl) * p.hq + h * p.G + g;
      uint2 packed;
      packed.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
      packed.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(p.out + row * kHeadDim + d0) = packed;
      if ((tid & 31) == 0) p.lse[row] = lse2 * 0.69314718055994531f;
    } else {
      const size_t row = static_cast<size_t>(slot) * p.rows_per_unit + r;
      *reinterpret_cast<float4*>(p.ws_o + row * kHeadDim + d0) =
          make_float4(acc[0] * inv, acc[1] * inv, acc[2] * inv, acc[3] * inv);
      if ((tid & 31) == 0) p.ws_lse[row] = lse2;
    }
  }
  named_barrier_sync(kBarConsumers, kWarps * 32);
}

__device__ __forceinline__ void run_consumer(const AttnParams& p, const Smem& sm, const Pipe& pipe, Cursor cu) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane >> 3, s8 = lane & 7;
  float qf[kCcRows][16];
  float o[kCcRows][16];
  float m_run[kCcRows], l_run[kCcRows];
  int stage = 0;
  uint32_t phase = 0;
  int piece_lt0 = 0;
  int anc_seq = -1;
  int consumed = 0;
  const int HR = p.hkv * p.row_blocks;

  for (; cu.t < cu.t_end; cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int h = cu.hr / p.row_blocks, rb = cu.hr - (cu.hr / p.row_blocks) * p.row_blocks;
    if (ti.first) {
      piece_lt0 = cu.lt;
#pragma unroll
      for (int r = 0; r < kCcRows; ++r) {
        const int rr = rb * p.rows_per_unit + r;
        uint4 a = make_uint4(0, 0, 0, 0), b = a;
        if (r < p.rows_per_unit && rr < p.rows_total) {
          const int nl = rr / p.G, g = rr - nl * p.G;
          const __nv_bfloat16* src =
              p.q + ((static_cast<size_t>(cu.c) * p.Nq + nl) * p.hq + h * p.G + g) * kHeadDim;
          a = *reinterpret_cast<const uint4*>(src + 8 * s8);
          b = *reinterpret_cast<const uint4*>(src + 64 + 8 * s8);
        }
        unpack16(a, b, qf[r]);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          qf[r][i] *= p.qscale;
          o[r][i] = 0.f;
        }
        m_run[r] = -INFINITY;
        l_run[r] = 0.f;
      }
    }
    if (ti.draft && p.tree) {
      const int seq = cu.c / (p.C / p.B);
      if (seq != anc_seq) {
        build_ancestor_masks(p, seq, sm.anc, sm.par, threadIdx.x, kWarps * 32, kBarConsumers);
        anc_seq = seq;
      }
    }
    // After a timed-out wait the warp keeps walking the tiles (so every named
    // barrier is still met) but waits for and computes nothing more.
    bool live = !*pipe.abort;
    if (live && !mbar_wait(smem_addr(&pipe.full[stage]), phase, p.err, p.wait_ns)) {
      *pipe.abort = 1;
      live = false;
    }
    live = __all_sync(0xffffffffu, live);  // the warp-wide MMA and shuffle steps below need the whole warp
    const uint32_t kbase = smem_addr(pipe.ring + static_cast<size_t>(stage) * kStageBytes);
    const uint32_t vbase = kbase + kKVTileBytes;
    const int kw0 = warp * kKeysPerWarp;
    if (live && kw0 < ti.nkeys) {
      float sc[kIters][kCcRows];
#pragma unroll
      for (int it = 0; it < kIters; ++it) {
        const int key = kw0 + it * 4 + grp;
        const uint4 ka = lds128(kbase + tile_off(key, s8));
        const uint4 kb = lds128(kbase + tile_off(key, 8 + s8));
        float kf[16];
        unpack16(ka, kb, kf);
#pragma unroll
        for (int r = 0; r < kCcRows; ++r) {
          float s = 0.f;
#pragma unroll
          for (int i = 0; i < 16; ++i) s = fmaf(qf[r][i], kf[i], s);
          s += __shfl_xor_sync(0xffffffffu, s, 1);
          s += __shfl_xor_sync(0xffffffffu, s, 2);
          s += __shfl_xor_sync(0xffffffffu, s, 4);
          bool valid = key < ti.nkeys;
          if (ti.draft) valid = valid && draft_visible(p, sm.anc, rb * p.rows_per_unit + r, ti.key0 + key);
          sc[it][r] = valid ? s : -INFINITY;
        }
      }
      float alpha[kCcRows], m_use[kCcRows];
      bool rescale = false;
#pragma unroll
      for (int r = 0; r < kCcRows; ++r) {
        float mx = sc[0][r];
#pragma unroll
        for (int it = 1; it < kIters; ++it) mx = fmaxf(mx, sc[it][r]);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float m_new = fmaxf(m_run[r], mx);
        m_use[r] = m_new == -INFINITY ? 0.f : m_new;
        alpha[r] = ex2(m_run[r] - m_use[r]);
        rescale |= m_new != m_run[r];
        m_run[r] = m_new;
      }
      if (rescale) {
#pragma unroll
        for (int r = 0; r < kCcRows; ++r) {
          l_run[r] *= alpha[r];
#pragma unroll
          for (int i = 0; i < 16; ++i) o[r][i] *= alpha[r];
        }
      }
#pragma unroll
      for (int it = 0; it < kIters; ++it) {
        const int key = kw0 + it * 4 + grp;
        float pr[kCcRows];
#pragma unroll
        for (int r = 0; r < kCcRows; ++r) {
          pr[r] = ex2(sc[it][r] - m_use[r]);
          l_run[r] += pr[r];
        }
        if (key < ti.nkeys) {  // rows past the tile's valid keys may hold NaN: never touch them
          const uint4 va = lds128(vbase + tile_off(key, s8));
          const uint4 vb = lds128(vbase + tile_off(key, 8 + s8));
          float vf[16];
          unpack16(va, vb, vf);
#pragma unroll
          for (int r = 0; r < kCcRows; ++r)
#pragma unroll
            for (int i = 0; i < 16; ++i) o[r][i] = fmaf(pr[r], vf[i], o[r][i]);
        }
      }
    }
    __syncwarp();
    if (live) {
      if (lane == 0) mbar_arrive(smem_addr(&pipe.empty[stage]));
      ++consumed;
    }
    if (++stage == kStages) {
      stage = 0;
      phase ^= 1u;
    }
    if (ti.last) {
      const bool whole = piece_lt0 == 0 && cu.lt == cu.ut - 1;
      const int slot = cu.c * HR + cu.hr + blockIdx.x;
      finalize(p, sm, cu.c, h, rb, slot, whole, o, m_run, l_run);
    }
  }
  if (threadIdx.x == 0) sm.misc[2] = consumed;
}

__global__ void __launch_bounds__(kThreads, 2)
    attn_cc_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ TensorMaps maps) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();  // the merge may be scheduled as CTAs finish
  const Smem sm = carve(smem_raw, p.C);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_addr(&sm.full[s]), 1);
      mbar_init(smem_addr(&sm.empty[s]), kWarps);
    }
    sm.misc[0] = 0;
    sm.misc[1] = 0;
    sm.misc[2] = 0;
    fence_mbar_init();
    prefetch_tensormap(&maps.tk);
    prefetch_tensormap(&maps.tv);
    prefetch_tensormap(&maps.dk);
    prefetch_tensormap(&maps.dv);
  }
  build_plan(p, sm.len, sm.base);  // contains __syncthreads
  // With KVSHOT_OVERLAP_PREVIOUS the kernel may have started before the preceding kernel ended:
  // q and the draft K/V (and every output) are touched only after it has.
  wait_for_prerequisite_grid();
  const Cursor cu = cursor_begin(p, sm.len, sm.base);
  Pipe pipe{sm.ring, sm.full, sm.empty, kStages, reinterpret_cast<volatile int*>(&sm.misc[0]), &sm.misc[1]};
  if (warp == kWarps) {
    run_producer(p, maps, pipe, sm.len, cu);
  } else {
    run_consumer(p, sm, pipe, cu);
  }
  __syncthreads();
  if (threadIdx.x == 0) drain_after_abort(p, pipe, sm.misc[2]);
}

}  // namespace

int attn_cc_ctas_per_sm() { return 2; }

size_t attn_cc_smem_bytes(int C) { return smem_bytes(C); }

cudaError_t attn_cc_occupancy(int C, int* ctas_per_sm) {
  const size_t smem = smem_bytes(C);
  cudaError_t e = cudaFuncSetAttribute(attn_cc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, attn_cc_kernel, kThreads, smem);
}

cudaError_t launch_attn_cc(const AttnParams& p, const TensorMaps& maps, bool pdl, cudaStream_t stream) {
  const size_t smem = smem_bytes(p.C);
  cudaError_t e = cudaFuncSetAttribute(attn_cc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch_maybe_pdl(attn_cc_kernel, dim3(p.num_ctas), dim3(kThreads), smem, pdl, stream, p, maps);
}

}  // namespace kvshot
