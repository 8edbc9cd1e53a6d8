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
// (KVSHOT_TARGET_FP8): the TMA brings each target tile's codes (128-byte rows,
// 128B-swizzled) into the upper half of its K and V tiles, and the consumer
// warps decode them straight into MMA fragments in registers; all MMAs run in
// f16 with the cache's power-of-two scales folded into the score scale and
// into P.  Fragment layouts of that variant: a lane's 16-byte load of one key
// row feeds four k-steps of S = Q K^T, so the head dimensions of q are taken
// in the same permuted order (k-step 4 kh + s, pair position 2 q4 -> dims
// 16 (2 q4 + kh) + 4 s + {0, 1}, position 8 + 2 q4 -> + {2, 3}); for O += P V a
// lane pairs the same 16 dims of two key rows with byte permutes, so the
// output columns are permuted too (n8 tile nd, column n -> dim 16 n + nd) and
// the write-out undoes it.  Draft tiles (bf16) are read into the same layouts
// and converted to f16 in registers.
//
// K/V tiles land in the halves layout (two 64-dim halves of 64 rows), or, for
// a bf16 paged cache, in the grouped layout (8-row groups holding both halves):
// there one TMA box brings a whole page of P < 64 tokens, or 8 draft slots,
// which halves the boxes per tile (Cfg's GR flag).
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

// 16 bytes from shared memory (ordered after the pipeline's barrier waits like the ldmatrix loads).
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

// Word t (0..3) of a 16-byte vector; t is a compile-time constant after unrolling.
__device__ __forceinline__ uint32_t word(const uint4& v, int t) {
  return t == 0 ? v.x : t == 1 ? v.y : t == 2 ? v.z : v.w;
}

// Byte offset, inside a K or V tile, of 16-byte chunk c (0..7: dims 16c .. 16c+15) of fp8 key row r:
// the codes occupy the tile's upper half as 128-byte rows under the TMA's 128-byte swizzle.
__device__ __forceinline__ uint32_t code_off(int r, int c) {
  return static_cast<uint32_t>(kHalfBytes + r * 128 + ((c ^ (r & 7)) << 4));
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

template <int MT, int KS, int STAGES, int MINB, bool F8 = false, bool GR = false>
struct Cfg {
  static constexpr bool kF8 = F8;                     // fp8 target tiles (KVSHOT_TARGET_FP8)
  static constexpr bool kGrouped = GR;                // every tile in the grouped layout (bf16 paged caches)
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
          if constexpr (CF::kF8) {
            // Permuted columns: o[nd][2i] is dim 32 q4 + nd, o[nd][2i + 1] dim 32 q4 + 16 + nd, so the
            // lane owns dims 32 q4 .. 32 q4 + 31 of the row and writes them as 16-byte vectors.
            if (whole) {
              const int nl = rr / p.G, gh = rr - nl * p.G;
              const size_t row = (static_cast<size_t>(c) * p.Nq + nl) * p.hq + h * p.G + gh;
              uint4* dst = reinterpret_cast<uint4*>(p.out + row * kHeadDim + 32 * q4);
#pragma unroll
              for (int hh = 0; hh < 2; ++hh)
#pragma unroll
                for (int v = 0; v < 2; ++v) {
                  const int e = 2 * i + hh, n0 = 8 * v;
                  dst[2 * hh + v] = make_uint4(pack_bf16x2(o[n0][e] * inv, o[n0 + 1][e] * inv),
                                               pack_bf16x2(o[n0 + 2][e] * inv, o[n0 + 3][e] * inv),
                                               pack_bf16x2(o[n0 + 4][e] * inv, o[n0 + 5][e] * inv),
                                               pack_bf16x2(o[n0 + 6][e] * inv, o[n0 + 7][e] * inv));
                }
              if (q4 == 0) p.lse[row] = lse2 * 0.69314718055994531f;
            } else {
              const size_t row = static_cast<size_t>(slot) * p.rows_per_unit + rl;
              float4* dst = reinterpret_cast<float4*>(p.ws_o + row * kHeadDim + 32 * q4);
#pragma unroll
              for (int hh = 0; hh < 2; ++hh)
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                  const int e = 2 * i + hh, n0 = 4 * v;
                  dst[4 * hh + v] = make_float4(o[n0][e] * inv, o[n0 + 1][e] * inv, o[n0 + 2][e] * inv,
                                                o[n0 + 3][e] * inv);
                }
              if (q4 == 0) p.ws_lse[row] = lse2;
            }
          } else if (whole) {
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
  int h = 0, rb = 0;  // KV head and row block of the current piece

  for (; cu.t < cu.t_end; cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int rl0 = mt * 16 + g;                       // rows of this thread within the unit
    if (ti.first) {
      h = cu.hr / p.row_blocks;
      rb = cu.hr - h * p.row_blocks;
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
          if constexpr (CF::kF8) {  // f16, k-step 4 kh + s on dims 16 (2 q4 + kh) + 4 s + {0..3}
            const int w = 8 * (2 * q4 + (kk >> 2)) + 2 * (kk & 3);
            qa[kk][i] = ok ? bf16x2_to_f16x2(src[w]) : 0u;
            qa[kk][2 + i] = ok ? bf16x2_to_f16x2(src[w + 1]) : 0u;
          } else {
            qa[kk][i] = ok ? src[kk * 8 + q4] : 0u;          // dims 16kk + 2q4, +1
            qa[kk][2 + i] = ok ? src[kk * 8 + 4 + q4] : 0u;  // dims 16kk + 8 + 2q4, +1
          }
        }
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
    if (live && !mbar_wait(smem_addr(&pipe.full[stage]), phase, p.err, p.wait_ns)) {
      *pipe.abort = 1;
      live = false;
    }
    live = __all_sync(0xffffffffu, live);  // the warp-wide MMA and shuffle steps below need the whole warp
    uint8_t* kptr = pipe.ring + static_cast<size_t>(stage) * kStageBytes;
    const uint32_t kbase = smem_addr(kptr);
    const uint32_t vbase = kbase + kKVTileBytes;
    const bool f16t = CF::kF8 && !ti.draft;  // this tile's K/V are fp8 codes (scaled by 2^exp)
    constexpr TileLayout lay = tile_layout(CF::kGrouped);
    if (!CF::kF8 && ti.nkeys < kTileKeys) {
      // V rows past the valid keys may be stale or NaN; the P.V product would
      // spread a NaN through 0 * NaN, so zero them (all consumer threads).  The
      // fp8 variant drops those rows in registers instead.
      if (live) {
        uint8_t* vptr = kptr + kKVTileBytes;
        const int nz = (kTileKeys - ti.nkeys) * 16;  // 16-byte chunks to clear
        for (int i = threadIdx.x; i < nz; i += CF::kWarps * 32) {
          const int key = ti.nkeys + (i >> 4), ch = i & 15;
          *reinterpret_cast<uint4*>(vptr + tile_off(key, ch, lay)) = make_uint4(0, 0, 0, 0);
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
      if constexpr (CF::kF8) {
        // Lane (g, q4) reads dims 16 (2 q4 + kh) .. + 15 of key row kw0 + 8j + g: four k-steps' B
        // fragments.  Under the swizzle the two rows of each 8-lane phase take chunks of opposite
        // parity, so the loads are free of bank conflicts.  Two accumulators per n8 tile (one per kh)
        // halve the MMA dependency chain.
        float s2[CF::kNT][4];
#pragma unroll
        for (int j = 0; j < CF::kNT; ++j) {
          s2[j][0] = s2[j][1] = s2[j][2] = s2[j][3] = 0.f;
          const int key = kw0 + j * 8 + g;
#pragma unroll
          for (int kh = 0; kh < 2; ++kh) {
            const int c = 2 * q4 + kh;
            uint32_t b[8];
            if (f16t) {
              const uint4 w = lds128(kbase + code_off(key, c));
              const uint2 f0 = e4m3x4_to_f16x4(w.x), f1 = e4m3x4_to_f16x4(w.y);
              const uint2 f2 = e4m3x4_to_f16x4(w.z), f3 = e4m3x4_to_f16x4(w.w);
              b[0] = f0.x; b[1] = f0.y; b[2] = f1.x; b[3] = f1.y;
              b[4] = f2.x; b[5] = f2.y; b[6] = f3.x; b[7] = f3.y;
            } else {
              const uint4 lo = lds128(kbase + tile_off(key, 2 * c, lay)), hi = lds128(kbase + tile_off(key, 2 * c + 1, lay));
              b[0] = bf16x2_to_f16x2(lo.x); b[1] = bf16x2_to_f16x2(lo.y);
              b[2] = bf16x2_to_f16x2(lo.z); b[3] = bf16x2_to_f16x2(lo.w);
              b[4] = bf16x2_to_f16x2(hi.x); b[5] = bf16x2_to_f16x2(hi.y);
              b[6] = bf16x2_to_f16x2(hi.z); b[7] = bf16x2_to_f16x2(hi.w);
            }
#pragma unroll
            for (int st = 0; st < 4; ++st) mma_f16_16816(kh ? s2[j] : s[j], qa[4 * kh + st], b[2 * st], b[2 * st + 1]);
          }
#pragma unroll
          for (int e = 0; e < 4; ++e) s[j][e] += s2[j][e];
        }
      } else {
#pragma unroll
        for (int j = 0; j < CF::kNT; ++j) {
          const int key = kw0 + j * 8 + lrow;
#pragma unroll
          for (int kp = 0; kp < 4; ++kp) {
            uint32_t b0, b1, b2, b3;
            ldmatrix_x4(kbase + tile_off(key, kp * 4 + lmat, lay), b0, b1, b2, b3);
            mma_bf16_16816(s[j], qa[2 * kp], b0, b1);
            mma_bf16_16816(s[j], qa[2 * kp + 1], b2, b3);
          }
        }
      }
      // Scale into the log2 domain, mask, row max over this warp's keys.
      const float qs = f16t ? p.qscale * p.k_scale : p.qscale;
      float mx[2] = {-INFINITY, -INFINITY};
      if (!ti.draft && ti.nkeys == kTileKeys) {  // a full prefix tile: every key is visible
#pragma unroll
        for (int j = 0; j < CF::kNT; ++j)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            s[j][e] *= qs;
            mx[e >> 1] = fmaxf(mx[e >> 1], s[j][e]);
          }
      } else {
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
        if constexpr (CF::kF8) {
          // B fragments from key rows kb, kb + 1 (b0) and kb + 8, kb + 9 (b1), dims 16g .. 16g + 15:
          // byte (or half-word) permutes pair the two rows' values of one dim, which lands in n8
          // tile nd = dim - 16g at column g.  Rows past the tile's valid keys read as zero.
          const int kb = kw0 + kk * 16 + 2 * q4;
          const int rows[4] = {kb, kb + 1, kb + 8, kb + 9};
          if (f16t) {
            uint4 w[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
              w[r] = lds128(vbase + code_off(rows[r], g));
              if (rows[r] >= ti.nkeys) w[r] = make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int t = 0; t < 4; ++t) {  // dims 16g + 4t .. 4t + 3 -> tiles 4t .. 4t + 3
              const uint2 ab0 = e4m3x4_to_f16x4(__byte_perm(word(w[0], t), word(w[1], t), 0x5140));
              const uint2 ab1 = e4m3x4_to_f16x4(__byte_perm(word(w[0], t), word(w[1], t), 0x7362));
              const uint2 cd0 = e4m3x4_to_f16x4(__byte_perm(word(w[2], t), word(w[3], t), 0x5140));
              const uint2 cd1 = e4m3x4_to_f16x4(__byte_perm(word(w[2], t), word(w[3], t), 0x7362));
              mma_f16_16816(o[4 * t], pa, ab0.x, cd0.x);
              mma_f16_16816(o[4 * t + 1], pa, ab0.y, cd0.y);
              mma_f16_16816(o[4 * t + 2], pa, ab1.x, cd1.x);
              mma_f16_16816(o[4 * t + 3], pa, ab1.y, cd1.y);
            }
          } else {
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {  // dims 16g + 8hh .. + 7 -> tiles 8hh .. 8hh + 7
              uint4 w[4];
#pragma unroll
              for (int r = 0; r < 4; ++r) {
                w[r] = lds128(vbase + tile_off(rows[r], 2 * g + hh, lay));
                if (rows[r] >= ti.nkeys) w[r] = make_uint4(0u, 0u, 0u, 0u);
              }
#pragma unroll
              for (int t = 0; t < 4; ++t) {  // word t: dims 16g + 8hh + 2t, +1 -> tiles 8hh + 2t, +1
                const uint32_t ab = word(w[0], t), bb = word(w[1], t), cb = word(w[2], t), db = word(w[3], t);
                mma_f16_16816(o[8 * hh + 2 * t], pa, bf16x2_to_f16x2(__byte_perm(ab, bb, 0x5410)),
                              bf16x2_to_f16x2(__byte_perm(cb, db, 0x5410)));
                mma_f16_16816(o[8 * hh + 2 * t + 1], pa, bf16x2_to_f16x2(__byte_perm(ab, bb, 0x7632)),
                              bf16x2_to_f16x2(__byte_perm(cb, db, 0x7632)));
              }
            }
          }
        } else {
          const int key = kw0 + kk * 16 + ((lmat & 1) << 3) + lrow;
#pragma unroll
          for (int ndp = 0; ndp < 8; ++ndp) {
            uint32_t b0, b1, b2, b3;
            ldmatrix_x4_trans(vbase + tile_off(key, 2 * ndp + (lmat >> 1), lay), b0, b1, b2, b3);
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

template <bool F8, bool GR = false> using Cfg1 = Cfg<1, 4, 3, 2, F8, GR>;
template <bool F8, bool GR = false> using Cfg2 = Cfg<2, 4, 4, 1, F8, GR>;
template <bool F8, bool GR = false> using Cfg3 = Cfg<3, 2, 4, 1, F8, GR>;
template <bool F8, bool GR = false> using Cfg4 = Cfg<4, 2, 4, 1, F8, GR>;

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

template <bool F8, bool GR>
cudaError_t launch_f8(const AttnParams& p, const TensorMaps& maps, int m_tiles, bool pdl, cudaStream_t stream) {
  switch (m_tiles) {
    case 1: return launch_cfg<Cfg1<F8, GR>>(p, maps, pdl, stream);
    case 2: return launch_cfg<Cfg2<F8, GR>>(p, maps, pdl, stream);
    case 3: return launch_cfg<Cfg3<F8, GR>>(p, maps, pdl, stream);
    case 4: return launch_cfg<Cfg4<F8, GR>>(p, maps, pdl, stream);
    default: return cudaErrorInvalidValue;
  }
}

// The grouped instantiations (p.prefix_grouped: bf16 paged caches) have the resources of the
// halves ones (same shared memory, registers capped by the same launch bounds), so the occupancy
// query above serves both.
cudaError_t launch_attn_mma(const AttnParams& p, const TensorMaps& maps, int m_tiles, bool pdl, cudaStream_t stream) {
  if (p.fp8) return launch_f8<true, false>(p, maps, m_tiles, pdl, stream);
  return p.prefix_grouped ? launch_f8<false, true>(p, maps, m_tiles, pdl, stream)
                          : launch_f8<false, false>(p, maps, m_tiles, pdl, stream);
}

}  // namespace kvshot
