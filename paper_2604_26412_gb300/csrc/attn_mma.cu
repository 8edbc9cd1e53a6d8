// attn_mma.cu -- draft attention for GQA stacks of 5..64 query rows per KV
// head (tree drafting: G heads x the draft nodes of one depth, or a whole
// draft chain), on the tensor cores with m16n8k16 bf16 MMAs.
//
// Each warp owns one 16-row m-tile of the stack and a slice of every key
// tile: S = Q K^T (Q fragments stay in registers for the whole piece, K
// fragments come from the 128B-swizzled TMA tile via ldmatrix), masked online
// softmax on the accumulator fragments, then O += P V with P re-packed from
// the S fragments and V fragments via ldmatrix.trans.  Math as in attn_cc.cu
// (Sec. 2.2 Eq. "kv-reattention" over M_i, Sec. 3.4 / App. B).
//
// A second instantiation (Cfg<..., true>) reads an fp8 e4m3 target cache
// (KVSHOT_TARGET_FP8): the TMA brings each target tile's codes into the upper
// half of its K and V tiles, the consumer warps expand every tile to f16 in
// shared memory, and all MMAs run in f16 with the cache's power-of-two scales
// folded into the score scale and into P.
#include <cuda_fp16.h>

#include "kvshot_attn_common.cuh"

namespace kvshot {
namespace {

using namespace dev;

// With an fp8 target cache (KVSHOT_TARGET_FP8) the kernel multiplies in f16: e4m3 -> f16 is exact
// (3 mantissa bits, exponents inside f16's range) and one conversion instruction per pair; q, the
// draft tiles and P are rounded to f16 (more mantissa than bf16; only values below 2^-14 lose
// bits).  The cache's power-of-two scales are folded into the score scale (keys) and into P
// (values), so one set of MMA fragments serves both kinds of tile.
// Four e4m3 codes (a 32-bit word, lowest byte first) -> four f16 values (two f16x2 words).
__device__ __forceinline__ uint2 e4m3x4_to_f16x4(uint32_t codes) {
  uint2 r;
  asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %2;\n\t"
      "cvt.rn.f16x2.e4m3x2 %0, lo;\n\tcvt.rn.f16x2.e4m3x2 %1, hi;\n\t}"
      : "=r"(r.x), "=r"(r.y)
      : "r"(codes));
  return r;
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t w) { return pack_f16x2(bf16_lo(w), bf16_hi(w)); }

__device__ __forceinline__ uint4 bf16x8_to_f16x8(uint4 v) {
  return make_uint4(bf16x2_to_f16x2(v.x), bf16x2_to_f16x2(v.y), bf16x2_to_f16x2(v.z), bf16x2_to_f16x2(v.w));
}

// 8 consecutive codes (dims 8ch .. 8ch+7 of one row) -> one 16-byte f16 chunk.
__device__ __forceinline__ uint4 expand8(const uint2 codes) {
  const uint2 lo = e4m3x4_to_f16x4(codes.x), hi = e4m3x4_to_f16x4(codes.y);
  return make_uint4(lo.x, lo.y, hi.x, hi.y);
}

// D += A * B, m16n8k16, f16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

constexpr int kBarConsumers = 1;
constexpr int kCombStride = kHeadDim + 4;  // padded fp32 row in the combine buffer

template <int MT, int KS, int STAGES, int MINB, bool F8 = false>
struct Cfg {
  static constexpr bool kF8 = F8;                     // fp8 target tiles (KVSHOT_TARGET_FP8)
  static constexpr int kMT = MT;                      // m16 tiles per unit
  static constexpr int kKS = KS;                      // key slices per tile
  static constexpr int kStages = STAGES;
  static constexpr int kMinBlocks = MINB;             // CTAs per SM the budget is sized for
  static constexpr int kWarps = MT * KS;              // consumer warps
  static constexpr int kThreads = (kWarps + 1) * 32;
  static constexpr int kKW = kTileKeys / KS;          // keys per warp per tile
  static constexpr int kNT = kKW / 8;                 // n8 tiles per warp per tile
  static constexpr int kRows = 16 * MT;               // rows per unit
};

struct Smem {
  uint8_t* ring;
  uint64_t* full;
  uint64_t* empty;
  uint64_t* anc;
  int* par;
  float* comb_o;   // [MT][16][kCombStride]
  float* comb_m;   // [KS][MT * 16]
  float* comb_l;   // [KS][MT * 16]
  int* misc;       // [0] abort, [1] issued, [2] consumed
  int* len;
  int* base;
};

template <class CF>
__host__ __device__ inline size_t smem_bytes(int C) {
  size_t off = static_cast<size_t>(CF::kStages) * kStageBytes;
  off += 2 * CF::kStages * sizeof(uint64_t);
  off += sizeof(uint64_t) * kMaxTreeNodes + sizeof(int) * kMaxTreeNodes;
  if (CF::kKS > 1) off += sizeof(float) * CF::kMT * 16 * kCombStride;  // only slices > 1 combine through smem
  off += 2 * sizeof(float) * CF::kKS * CF::kRows;
  off += sizeof(int) * 4;
  off += sizeof(int) * (2 * C + 1);
  return off + 1024;
}

template <class CF>
__device__ Smem carve(uint8_t* raw, int C) {
  Smem s;
  uint8_t* p = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  s.ring = p;
  p += CF::kStages * kStageBytes;
  s.full = reinterpret_cast<uint64_t*>(p);
  s.empty = s.full + CF::kStages;
  s.anc = s.empty + CF::kStages;
  s.par = reinterpret_cast<int*>(s.anc + kMaxTreeNodes);
  s.comb_o = reinterpret_cast<float*>(s.par + kMaxTreeNodes);
  s.comb_m = s.comb_o + (CF::kKS > 1 ? CF::kMT * 16 * kCombStride : 0);
  s.comb_l = s.comb_m + CF::kKS * CF::kRows;
  s.misc = reinterpret_cast<int*>(s.comb_l + CF::kKS * CF::kRows);
  s.len = s.misc + 4;
  s.base = s.len + C;
  return s;
}

// Combine the KS key-slice warps of each m-tile and write the piece: the
// final bf16 output + lse if the piece is the whole unit, else the
// normalised fp32 partial + log2-domain lse into workspace slot `slot`.
template <class CF>
__device__ __forceinline__ void finalize(const AttnParams& p, const Smem& sm, int c, int h, int rb, int slot, bool whole,
                         float (&o)[16][4], const float (&m_run)[2], float (&l_run)[2]) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = warp % CF::kMT, ks = warp / CF::kMT;
  const int g = lane >> 2, q4 = lane & 3;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 1);
    l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 2);
  }
  const int row0 = mt * 16 + g;  // this thread's rows: row0 and row0 + 8
  if (q4 == 0) {
    sm.comb_m[ks * CF::kRows + row0] = m_run[0];
    sm.comb_m[ks * CF::kRows + row0 + 8] = m_run[1];
    sm.comb_l[ks * CF::kRows + row0] = l_run[0];
    sm.comb_l[ks * CF::kRows + row0 + 8] = l_run[1];
  }
  named_barrier_sync(kBarConsumers, CF::kWarps * 32);
  float M[2], Lsum[2], wself[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = row0 + 8 * i;
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < CF::kKS; ++k) mx = fmaxf(mx, sm.comb_m[k * CF::kRows + row]);
    M[i] = mx;
    float Ls = 0.f;
    if (mx != -INFINITY) {
#pragma unroll
      for (int k = 0; k < CF::kKS; ++k) {
        const float mk = sm.comb_m[k * CF::kRows + row];
        Ls += (mk == -INFINITY ? 0.f : ex2(mk - mx)) * sm.comb_l[k * CF::kRows + row];
      }
    }
    Lsum[i] = Ls;
    wself[i] = (m_run[i] == -INFINITY || mx == -INFINITY) ? 0.f : ex2(m_run[i] - mx);
  }
#pragma unroll
  for (int nd = 0; nd < 16; ++nd) {
    o[nd][0] *= wself[0];
    o[nd][1] *= wself[0];
    o[nd][2] *= wself[1];
    o[nd][3] *= wself[1];
  }
  float* buf = sm.comb_o + mt * 16 * kCombStride;
  // Key slices accumulate into the buffer one after another; the last one writes out.
#pragma unroll
  for (int k = 0; k < CF::kKS; ++k) {
    if (ks == k) {
      if (k > 0) {
#pragma unroll
        for (int nd = 0; nd < 16; ++nd) {
          const float2 a = *reinterpret_cast<const float2*>(buf + g * kCombStride + nd * 8 + 2 * q4);
          const float2 b = *reinterpret_cast<const float2*>(buf + (g + 8) * kCombStride + nd * 8 + 2 * q4);
          o[nd][0] += a.x;
          o[nd][1] += a.y;
          o[nd][2] += b.x;
          o[nd][3] += b.y;
        }
      }
      if (k < CF::kKS - 1) {
#pragma unroll
        for (int nd = 0; nd < 16; ++nd) {
          *reinterpret_cast<float2*>(buf + g * kCombStride + nd * 8 + 2 * q4) = make_float2(o[nd][0], o[nd][1]);
          *reinterpret_cast<float2*>(buf + (g + 8) * kCombStride + nd * 8 + 2 * q4) =
              make_float2(o[nd][2], o[nd][3]);
        }
      } else {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const int rl = row0 + 8 * i;                 // row within this unit (row block)
          const int rr = rb * p.rows_per_unit + rl;    // row within the GQA stack
          if (rl >= p.rows_per_unit || rr >= p.rows_total) continue;
          const float inv = Lsum[i] > 0.f ? 1.f / Lsum[i] : 0.f;
          const float lse2 = Lsum[i] > 0.f ? M[i] + __log2f(Lsum[i]) : -INFINITY;
          if (whole) {
            const int nl = rr / p.G, gh = rr - nl * p.G;
            const size_t row = (static_cast<size_t>(c) * p.Nq + nl) * p.hq + h * p.G + gh;
            __nv_bfloat16* dst = p.out + row * kHeadDim + 2 * q4;
#pragma unroll
            for (int nd = 0; nd < 16; ++nd)
              *reinterpret_cast<uint32_t*>(dst + nd * 8) = pack_bf16x2(o[nd][2 * i] * inv, o[nd][2 * i + 1] * inv);
            if (q4 == 0) p.lse[row] = lse2 * 0.69314718055994531f;
          } else {
            const size_t row = static_cast<size_t>(slot) * p.rows_per_unit + rl;
            float* dst = p.ws_o + row * kHeadDim + 2 * q4;
#pragma unroll
            for (int nd = 0; nd < 16; ++nd)
              *reinterpret_cast<float2*>(dst + nd * 8) = make_float2(o[nd][2 * i] * inv, o[nd][2 * i + 1] * inv);
            if (q4 == 0) p.ws_lse[row] = lse2;
          }
        }
      }
    }
    if (k < CF::kKS - 1) named_barrier_sync(kBarConsumers, CF::kWarps * 32);
  }
  named_barrier_sync(kBarConsumers, CF::kWarps * 32);
}

template <class CF>
__device__ __forceinline__ void run_consumer(const AttnParams& p, const Smem& sm, const Pipe& pipe, Cursor cu) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = warp % CF::kMT, ks = warp / CF::kMT;
  const int g = lane >> 2, q4 = lane & 3;
  const int HR = p.hkv * p.row_blocks;
  uint32_t qa[8][4];  // bf16 pairs, or f16 pairs in the fp8 variant
  float o[16][4];
  float m_run[2], l_run[2];
  int stage = 0;
  uint32_t phase = 0;
  int piece_lt0 = 0, anc_seq = -1, consumed = 0;

  for (; cu.t < cu.t_end; cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int h = cu.hr / p.row_blocks, rb = cu.hr - (cu.hr / p.row_blocks) * p.row_blocks;
    const int rl0 = mt * 16 + g;                       // rows of this thread within the unit
    if (ti.first) {
      piece_lt0 = cu.lt;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int rl = rl0 + 8 * i, rr = rb * p.rows_per_unit + rl;
        const bool ok = rl < p.rows_per_unit && rr < p.rows_total;
        const int nl = ok ? rr / p.G : 0, gh = ok ? rr - nl * p.G : 0;
        const uint32_t* src = reinterpret_cast<const uint32_t*>(
            p.q + ((static_cast<size_t>(cu.c) * p.Nq + nl) * p.hq + h * p.G + gh) * kHeadDim);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          qa[kk][i] = ok ? src[kk * 8 + q4] : 0u;          // dims 16kk + 2q4, +1
          qa[kk][2 + i] = ok ? src[kk * 8 + 4 + q4] : 0u;  // dims 16kk + 8 + 2q4, +1
        }
      }
      if constexpr (CF::kF8) {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
#pragma unroll
          for (int r = 0; r < 4; ++r) qa[kk][r] = bf16x2_to_f16x2(qa[kk][r]);
      }
#pragma unroll
      for (int nd = 0; nd < 16; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
      m_run[0] = m_run[1] = -INFINITY;
      l_run[0] = l_run[1] = 0.f;
    }
    if (ti.draft && p.tree) {
      const int seq = cu.c / (p.C / p.B);
      if (seq != anc_seq) {
        build_ancestor_masks(p, seq, sm.anc, sm.par, threadIdx.x, CF::kWarps * 32, kBarConsumers);
        anc_seq = seq;
      }
    }
    bool live = !*pipe.abort;
    if (live && !mbar_wait(smem_addr(&pipe.full[stage]), phase, p.err)) {
      *pipe.abort = 1;
      live = false;
    }
    uint8_t* kptr = pipe.ring + static_cast<size_t>(stage) * kStageBytes;
    const uint32_t kbase = smem_addr(kptr);
    const uint32_t vbase = kbase + kKVTileBytes;
    const bool f16t = CF::kF8 && !ti.draft;  // this tile's K/V are fp8 codes (scaled by 2^exp)
    if constexpr (CF::kF8) {
      // fp8 variant: every tile becomes f16 in place.  Target tiles: the e4m3 rows (128 bytes per
      // key) sit in the upper half of the K and V tiles; a row's upper f16 half lands exactly on that
      // row's codes, which the 16 lanes converting the row have all loaded before the warp stores.
      // Draft tiles: each 16-byte chunk of 8 bf16 is rewritten as 8 f16.  With one m-tile per unit
      // each warp reads only the K and V rows of its own key slice, so it converts just those and
      // no barrier is needed (except before the tail rows are zeroed).
      constexpr bool kOwnRows = CF::kMT == 1;
      const int row0 = kOwnRows ? ks * CF::kKW : 0;            // first key row this warp converts
      const int nrows = kOwnRows ? CF::kKW : kTileKeys;        // key rows per K (and per V) tile
      const int w0 = kOwnRows ? 0 : warp, wstep = kOwnRows ? 1 : CF::kWarps;
      if (__all_sync(0xffffffffu, live)) {
        if (f16t) {
          // Two rows per warp instruction: lane = (row parity, 16-byte chunk ch) takes the row's codes
          // 8ch .. 8ch+7, so the 16 lanes of a row read it whole (8 bytes each) and write its 16
          // chunks, which the 128-byte swizzle spreads over all banks.
          for (int g2 = w0; g2 < nrows; g2 += wstep) {
            const int r = g2 * 2 + (lane >> 4);  // K rows, then V rows
            const int kv = r / nrows, key = row0 + r % nrows, ch = lane & 15;
            uint8_t* tile = kptr + kv * kKVTileBytes;
            const uint2 codes = *reinterpret_cast<const uint2*>(tile + kHalfBytes + key * 128 + ch * 8);
            __syncwarp();
            *reinterpret_cast<uint4*>(tile + tile_off(key, ch)) = expand8(codes);
          }
        } else {
          for (int i = w0 * 32 + lane; i < 2 * nrows * 16; i += wstep * 32) {
            const int r = i / 16, ch = i % 16;
            uint4* chunk =
                reinterpret_cast<uint4*>(kptr + (r / nrows) * kKVTileBytes + tile_off(row0 + r % nrows, ch));
            *chunk = bf16x8_to_f16x8(*chunk);
          }
        }
        fence_proxy_async_smem();  // the next TMA write into this stage comes after these stores
      }
      if (!kOwnRows || ti.nkeys < kTileKeys) named_barrier_sync(kBarConsumers, CF::kWarps * 32);
    }
    if (ti.nkeys < kTileKeys) {
      // V rows past the valid keys may be stale or NaN; the P.V product would
      // spread a NaN through 0 * NaN, so zero them (all consumer threads).
      if (live) {
        uint8_t* vptr = kptr + kKVTileBytes;
        const int nz = (kTileKeys - ti.nkeys) * 16;  // 16-byte chunks to clear
        for (int i = threadIdx.x; i < nz; i += CF::kWarps * 32) {
          const int key = ti.nkeys + (i >> 4), ch = i & 15;
          *reinterpret_cast<uint4*>(vptr + tile_off(key, ch)) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
      }
      named_barrier_sync(kBarConsumers, CF::kWarps * 32);
    }
    const int kw0 = ks * CF::kKW;
    if (live && kw0 < ti.nkeys) {
      float s[CF::kNT][4];
#pragma unroll
      for (int j = 0; j < CF::kNT; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
      const int lrow = lane & 7, lmat = lane >> 3;
#pragma unroll
      for (int j = 0; j < CF::kNT; ++j) {
        const int key = kw0 + j * 8 + lrow;
#pragma unroll
        for (int kp = 0; kp < 4; ++kp) {
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4(kbase + tile_off(key, kp * 4 + lmat), b0, b1, b2, b3);
          if constexpr (CF::kF8) {
            mma_f16_16816(s[j], qa[2 * kp], b0, b1);
            mma_f16_16816(s[j], qa[2 * kp + 1], b2, b3);
          } else {
            mma_bf16_16816(s[j], qa[2 * kp], b0, b1);
            mma_bf16_16816(s[j], qa[2 * kp + 1], b2, b3);
          }
        }
      }
      // Scale into the log2 domain, mask, row max over this warp's keys.
      const float qs = f16t ? p.qscale * p.k_scale : p.qscale;
      float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int j = 0; j < CF::kNT; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kw0 + j * 8 + 2 * q4 + (e & 1);
          const int rl = rl0 + (e >> 1) * 8;
          bool valid = key < ti.nkeys;
          if (ti.draft) valid = valid && draft_visible(p, sm.anc, rb * p.rows_per_unit + rl, ti.key0 + key);
          s[j][e] = valid ? s[j][e] * qs : -INFINITY;
          mx[e >> 1] = fmaxf(mx[e >> 1], s[j][e]);
        }
      }
      float alpha[2], m_use[2];
      bool rescale = false;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
        mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
        const float m_new = fmaxf(m_run[i], mx[i]);
        m_use[i] = m_new == -INFINITY ? 0.f : m_new;
        alpha[i] = ex2(m_run[i] - m_use[i]);
        rescale |= m_new != m_run[i];
        m_run[i] = m_new;
      }
      if (__any_sync(0xffffffffu, rescale)) {
        l_run[0] *= alpha[0];
        l_run[1] *= alpha[1];
#pragma unroll
        for (int nd = 0; nd < 16; ++nd) {
          o[nd][0] *= alpha[0];
          o[nd][1] *= alpha[0];
          o[nd][2] *= alpha[1];
          o[nd][3] *= alpha[1];
        }
      }
#pragma unroll
      for (int j = 0; j < CF::kNT; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          s[j][e] = ex2(s[j][e] - m_use[e >> 1]);
          l_run[e >> 1] += s[j][e];
        }
      }
      // O += P V, 16 keys per k-step.
#pragma unroll
      for (int kk = 0; kk < CF::kNT / 2; ++kk) {
        uint32_t pa[4];
        if constexpr (CF::kF8) {  // P times the value scale, in f16 (the running sum keeps the unscaled P)
          const float vs = f16t ? p.v_scale : 1.f;
          pa[0] = pack_f16x2(s[2 * kk][0] * vs, s[2 * kk][1] * vs);
          pa[1] = pack_f16x2(s[2 * kk][2] * vs, s[2 * kk][3] * vs);
          pa[2] = pack_f16x2(s[2 * kk + 1][0] * vs, s[2 * kk + 1][1] * vs);
          pa[3] = pack_f16x2(s[2 * kk + 1][2] * vs, s[2 * kk + 1][3] * vs);
        } else {
          pa[0] = pack_bf16x2(s[2 * kk][0], s[2 * kk][1]);
          pa[1] = pack_bf16x2(s[2 * kk][2], s[2 * kk][3]);
          pa[2] = pack_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
          pa[3] = pack_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
        }
        const int key = kw0 + kk * 16 + ((lmat & 1) << 3) + lrow;
#pragma unroll
        for (int ndp = 0; ndp < 8; ++ndp) {
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4_trans(vbase + tile_off(key, 2 * ndp + (lmat >> 1)), b0, b1, b2, b3);
          if constexpr (CF::kF8) {
            mma_f16_16816(o[2 * ndp], pa, b0, b1);
            mma_f16_16816(o[2 * ndp + 1], pa, b2, b3);
          } else {
            mma_bf16_16816(o[2 * ndp], pa, b0, b1);
            mma_bf16_16816(o[2 * ndp + 1], pa, b2, b3);
          }
        }
      }
    }
    __syncwarp();
    if (live) {
      if (lane == 0) mbar_arrive(smem_addr(&pipe.empty[stage]));
      ++consumed;
    }
    if (++stage == CF::kStages) {
      stage = 0;
      phase ^= 1u;
    }
    if (ti.last) {
      const bool whole = piece_lt0 == 0 && cu.lt == cu.ut - 1;
      const int slot = cu.c * HR + cu.hr + blockIdx.x;
      finalize<CF>(p, sm, cu.c, h, rb, slot, whole, o, m_run, l_run);
    }
  }
  if (threadIdx.x == 0) sm.misc[2] = consumed;
}

template <class CF>
__global__ void __launch_bounds__(CF::kThreads, CF::kMinBlocks)
    attn_mma_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ TensorMaps maps) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();  // the merge may be scheduled as CTAs finish
  const Smem sm = carve<CF>(smem_raw, p.C);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int s = 0; s < CF::kStages; ++s) {
      mbar_init(smem_addr(&sm.full[s]), 1);
      mbar_init(smem_addr(&sm.empty[s]), CF::kWarps);
    }
    sm.misc[0] = sm.misc[1] = sm.misc[2] = 0;
    fence_mbar_init();
    prefetch_tensormap(&maps.tk);
    prefetch_tensormap(&maps.tv);
    prefetch_tensormap(&maps.dk);
    prefetch_tensormap(&maps.dv);
  }
  build_plan(p, sm.len, sm.base);
  // With KVSHOT_OVERLAP_PREVIOUS the kernel may have started before the preceding kernel ended:
  // q and the draft K/V (and every output) are touched only after it has.
  wait_for_prerequisite_grid();
  const Cursor cu = cursor_begin(p, sm.len, sm.base);
  Pipe pipe{sm.ring, sm.full, sm.empty, CF::kStages, reinterpret_cast<volatile int*>(&sm.misc[0]), &sm.misc[1]};
  if (warp == CF::kWarps) {
    run_producer(p, maps, pipe, sm.len, cu);
  } else {
    run_consumer<CF>(p, sm, pipe, cu);
  }
  __syncthreads();
  if (threadIdx.x == 0) drain_after_abort(p, pipe, sm.misc[2]);
}

template <bool F8> using Cfg1 = Cfg<1, 4, 3, 2, F8>;
template <bool F8> using Cfg2 = Cfg<2, 4, 4, 1, F8>;
template <bool F8> using Cfg3 = Cfg<3, 2, 4, 1, F8>;
template <bool F8> using Cfg4 = Cfg<4, 2, 4, 1, F8>;

template <class CF>
cudaError_t launch_cfg(const AttnParams& p, const TensorMaps& maps, bool pdl, cudaStream_t stream) {
  const size_t smem = smem_bytes<CF>(p.C);
  cudaError_t e = cudaFuncSetAttribute(attn_mma_kernel<CF>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch_maybe_pdl(attn_mma_kernel<CF>, dim3(p.num_ctas), dim3(CF::kThreads), smem, pdl, stream, p, maps);
}

template <class CF>
cudaError_t occupancy_cfg(int C, int* ctas) {
  const size_t smem = smem_bytes<CF>(C);
  cudaError_t e = cudaFuncSetAttribute(attn_mma_kernel<CF>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas, attn_mma_kernel<CF>, CF::kThreads, smem);
}

}  // namespace

int attn_mma_ctas_per_sm(int m_tiles) { return m_tiles == 1 ? Cfg1<false>::kMinBlocks : 1; }

template <bool F8>
cudaError_t occupancy_f8(int m_tiles, int C, int* ctas_per_sm) {
  switch (m_tiles) {
    case 1: return occupancy_cfg<Cfg1<F8>>(C, ctas_per_sm);
    case 2: return occupancy_cfg<Cfg2<F8>>(C, ctas_per_sm);
    case 3: return occupancy_cfg<Cfg3<F8>>(C, ctas_per_sm);
    case 4: return occupancy_cfg<Cfg4<F8>>(C, ctas_per_sm);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t attn_mma_occupancy(int m_tiles, int C, bool fp8, int* ctas_per_sm) {
  return fp8 ? occupancy_f8<true>(m_tiles, C, ctas_per_sm) : occupancy_f8<false>(m_tiles, C, ctas_per_sm);
}

template <bool F8>
cudaError_t launch_f8(const AttnParams& p, const TensorMaps& maps, int m_tiles, bool pdl, cudaStream_t stream) {
  switch (m_tiles) {
    case 1: return launch_cfg<Cfg1<F8>>(p, maps, pdl, stream);
    case 2: return launch_cfg<Cfg2<F8>>(p, maps, pdl, stream);
    case 3: return launch_cfg<Cfg3<F8>>(p, maps, pdl, stream);
    case 4: return launch_cfg<Cfg4<F8>>(p, maps, pdl, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_attn_mma(const AttnParams& p, const TensorMaps& maps, int m_tiles, bool pdl, cudaStream_t stream) {
  return p.fp8 ? launch_f8<true>(p, maps, m_tiles, pdl, stream) : launch_f8<false>(p, maps, m_tiles, pdl, stream);
}

}  // namespace kvshot
