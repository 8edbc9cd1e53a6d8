// attn_tc.cu -- draft attention on the 5th-generation tensor cores (tcgen05),
// accumulators in tensor memory (TMEM).
//
// Per unit (cache, KV head, block of up to 128 stacked GQA rows), per 64-key
// tile (Sec. 2.2 Eq. "kv-reattention" over the memory M_i of Sec. 3.4 /
// App. B, as an online softmax in the log2 domain):
//   S = Q K^T      tcgen05.mma M=128 N=64  K=128 (8 x K16), A = Q (smem), B = K tile (smem), D = S (TMEM)
//   P = softmax(S) TMEM -> registers -> bf16 pairs written back over the S columns (TMEM)
//   O += P V       tcgen05.mma M=128 N=128 K=64 (4 x K16), A = P (TMEM), B = V tile (smem, MN-major), D = O (TMEM)
// Warp roles: warps 0..7 are two softmax warpgroups; warps 10 and 9 load the
// K and V tiles of even and odd tiles by TMA, warp 9 also the q blocks (a
// single warp keeps too few bulk-tensor loads in flight to reach full HBM
// bandwidth); warp 11 owns TMEM and one of its threads issues every QK^T, one
// thread of warp 8 every P.V.
// Row modes (one kernel each):
//  - dense (up to 128 rows, a thread per TMEM lane) and spread (up to 64 rows,
//    16 per TMEM lane quarter, two threads per row): warpgroup w owns the tiles
//    t with t % 2 == w, with its own running max/sum and its own O_w, so the
//    two warpgroups' per-tile chains overlap; their states are merged by
//    log-sum-exp at the end of each piece.  Four S buffers; an S buffer is
//    free again when P.V of its tile completes.
//  - paired (129..256 rows, attn_tc_pair_kernel): two 128-row blocks per unit,
//    warpgroup w owning block w on every tile, so each K/V tile is read once
//    for both.  14 warps: block 1 has QK^T and P.V issuers of its own (warps
//    12, 13), so the two blocks' dependent MMA chains overlap in the tensor
//    pipe and each block's commit waits for its own chain only.
// O_w is rescaled in TMEM only when a row's running max grows by more than
// 2^8 (lazy rescale).  Rows of the 128-row MMA that hold no stacked row carry
// no output.
// K and V tiles are staged in the grouped layout (kGroupBytes): one TMA box
// brings a whole page of up to 64 tokens with both 64-dim halves, so a tile of
// 16-token pages takes 4 boxes per tensor instead of 8.  Ring depths (5 K,
// 6 V) were measured on GB300: the bytes in flight per SM that the rings
// allow bound how fast one CTA streams.
// fp8 target cache (dense and spread rows; the default for 17..128 rows): the
// producer warps land the e4m3 codes of each tile in a landing slot, and the
// softmax warpgroup between tiles decodes them into the f16 K and V ring tiles
// (three tiles ahead of the tile it takes next); q and the draft tiles are
// converted to f16 by the producers and the MMAs multiply in f16.
#include <cuda_fp16.h>

#include "kvshot_attn_common.cuh"
#include "kvshot_tcgen05.cuh"

namespace kvshot {
namespace {

using namespace dev;
using namespace tc;

constexpr int kNK = 5;                     // K tiles in flight (freed when QK^T completes)
constexpr int kNV = 6;                     // V tiles in flight (freed when P.V completes)
constexpr int kKVBytes = kKVTileBytes;     // one K or V tile
constexpr int kNS = 4;                     // S buffers in TMEM: QK^T may run up to 4 tiles ahead of P.V
constexpr int kThreads = 12 * 32;
constexpr int kProducerWarp = 10;          // K and V loads of even tiles
constexpr int kProducerVWarp = 9;          // K and V loads of odd tiles, q blocks
constexpr int kMmaWarp = 11;               // TMEM owner, QK^T issuer
constexpr int kMmaPvWarp = 8;              // P.V issuer
constexpr int kSoftmaxThreads = 256;       // two warpgroups
constexpr int kBarSoftmax = 1;             // named barrier among the softmax warps
constexpr uint32_t kTmemCols = 512;        // S0..S3 [0,256), O0 [256,384), O1 [384,512)
constexpr uint32_t kTmemO = kNS * kTileKeys;
constexpr int kMiscInts = 22;
// fp8 (e4m3) target cache: rings of f16 tiles, decoded by the softmax warpgroups from landing slots
// that the producer warps fill (8 KB of K codes and 8 KB of V codes each).
constexpr int kF8NK = 3;
constexpr int kF8NV = 4;
constexpr int kLandBytes = 2 * kTileKeys * 128;  // one landing slot: a tile's K codes then its V codes
constexpr int kLandSlots = 4;                    // tile t lands in slot t % kLandSlots, freed when it is decoded
constexpr int kDecodeAhead = 3;                  // the softmax warpgroup done with tile t decodes tile t + 3
constexpr int kBarDecode0 = 2;                   // named barriers 2, 3: the 128 threads of warpgroup 0, 1
static_assert(kLandSlots % 2 == 0, "a landing slot must stay with one producer warp (t and t - kLandSlots)");
constexpr float kRescaleThreshold = 8.0f;  // log2 units: rescale O when the max grows by > 256x

// Row modes.  Dense: one block of up to 128 stacked rows, one thread per TMEM lane, the two
// warpgroups alternating tiles.  Spread: up to 64 rows, 16 per TMEM lane quarter.  Pair: two
// 128-row blocks of one KV head (129..256 rows), warpgroup w owning block w on every tile.
constexpr int kModeDense = 0, kModeSpread = 1, kModePair = 2;
constexpr int kPairThreads = 14 * 32;      // paired blocks: warps 12 and 13 issue QK^T and P.V of block 1
constexpr int kMmaWarp1 = 12;              // paired blocks: QK^T issuer of block 1
constexpr int kMmaPvWarp1 = 13;            // paired blocks: P.V issuer of block 1
constexpr int kPairNK = 4;                 // paired blocks: K tiles in flight
constexpr int kPairNV = 5;                 // paired blocks: V tiles in flight
template <int M>
struct RingOf {
  static constexpr int NK = M == kModePair ? kPairNK : kNK;
  static constexpr int NV = M == kModePair ? kPairNV : kNV;
};

__device__ __forceinline__ uint32_t pack_f16x2_tc(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Two-lane fp32 FMA and add (one instruction each on sm_100 and later).
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

// Row maximum of N raw scores (four independent chains of three-input maxima).
template <int N>
__device__ __forceinline__ float row_max(const float (&s)[N]) {
  float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int k = 0; k < N / 2; ++k) m4[k & 3] = max3(m4[k & 3], s[2 * k], s[2 * k + 1]);
  return fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
}

// P = 2^(s qs - m) of N raw scores (qs > 0), packed in pairs into pk (bf16, or f16 times vs), and the
// sum of the unrounded values.  The scale rides in the exponent's FMA, two lanes per instruction.
template <int N, bool kF16>
__device__ __forceinline__ float row_exp(const float (&s)[N], float qs, float m, float vs, uint32_t (&pk)[N / 2]) {
  const float2 q2 = make_float2(qs, qs), nm2 = make_float2(-m, -m);
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < N / 2; ++k) {
    const float2 x = fma2(make_float2(s[2 * k], s[2 * k + 1]), q2, nm2);
    const float2 e = make_float2(ex2(x.x), ex2(x.y));
    if (k & 1) acc1 = add2(acc1, e);
    else acc0 = add2(acc0, e);
    if constexpr (kF16) pk[k] = pack_f16x2_tc(e.x * vs, e.y * vs);
    else pk[k] = pack_bf16x2(e.x, e.y);
  }
  return (acc0.x + acc0.y) + (acc1.x + acc1.y);
}

// A buffer of bf16 values (whole 16-byte chunks, shared-memory address `buf`) converted in place to f16
// by one warp: exact for magnitudes in [2^-14, 65504] (values below 2^-14 lose low bits).  The layout
// (swizzle included) is kept, since every element stays where it was.
__device__ __forceinline__ void bf16_to_f16_inplace(uint32_t buf, int bytes, int lane) {
#pragma unroll 4
  for (int off = lane * 16; off < bytes; off += 32 * 16) {
    uint4 v = lds128(buf + off);
    v.x = pack_f16x2_tc(bf16_lo(v.x), bf16_hi(v.x));
    v.y = pack_f16x2_tc(bf16_lo(v.y), bf16_hi(v.y));
    v.z = pack_f16x2_tc(bf16_lo(v.z), bf16_hi(v.z));
    v.w = pack_f16x2_tc(bf16_lo(v.w), bf16_hi(v.w));
    sts128(buf + off, v);
  }
}

// Byte offset of 16-byte chunk `ch` (dims 8ch..8ch+7) of key r in a K or V
// tile of either layout (128-byte swizzle: chunk index XOR row index mod 8).
__device__ __forceinline__ uint32_t tile_off_tc(int r, int ch, bool grouped) {
  const uint32_t sw = static_cast<uint32_t>(((ch & 7) ^ (r & 7)) << 4);
  if (grouped) return static_cast<uint32_t>((r >> 3) * kGroupBytes + (ch >> 3) * kGroupHalfBytes + (r & 7) * 128) + sw;
  return static_cast<uint32_t>((ch >> 3) * kHalfBytes + r * 128) + sw;
}

// ------------------------------------------------------------ shared memory

struct Smem {
  uint8_t* kring;      // kNK x K tile
  uint8_t* vring;      // kNV x V tile
  uint8_t* qbuf;       // one q block
  uint8_t* land;       // fp8 cache: [kLandSlots] landing slots of e4m3 codes (K codes, then V codes)
  uint64_t* kfull;     // [kNK]  TMA -> MMA
  uint64_t* kempty;    // [kNK]  QK^T of the slot's tile completed -> TMA
  uint64_t* vfull;     // [kNV]  TMA -> MMA, softmax
  uint64_t* vempty;    // [kNV]  P.V completion -> TMA
  uint64_t* qfull;     // [1]
  uint64_t* qempty;    // [1]
  uint64_t* sfull;     // [kNS]  S buffer written (QK^T completion)
  uint64_t* sfree;     // [kNS]  P.V of the tile in the S buffer completed: the buffer is free
  uint64_t* pfull;     // [kNS]  P written over the S buffer (the owning warpgroup's 128 threads)
  uint64_t* ofree;     // [1]  epilogue finished reading O
  uint64_t* mmadone;   // [2]  every QK^T / every P.V completed
  uint64_t* lfull;     // fp8 cache: [kLandSlots] the tile's codes landed (TMA), or a draft tile passed through
  uint64_t* lfree;     // fp8 cache: [kLandSlots] the tile in the slot was decoded: the slot is free
  uint64_t* qland;     // fp8 cache: [1] bf16 q block landed (converted to f16 before qfull)
  uint64_t* dland;     // fp8 cache: [2] a producer warp's bf16 draft tile landed (converted before kfull / vfull)
  uint64_t* anc;       // [64]
  int* par;            // [64]
  float* comb;         // [128][2] second warpgroup's (max, sum) per row at a piece end
  uint32_t* tmem_base;
  int* misc;           // [0] abort, [2] K tiles consumed, [3]/[4] q blocks issued/consumed, [6] V tiles consumed,
                       // [8..9] / [10..11] K / V tiles issued per producer warp, [12..13] fp8: tiles of
                       // parity 0 / 1 whose landing was issued, [14..15] fp8: of those, tiles whose landing a
                       // decoder waited, [1] fp8: q blocks converted, [16..17] / [18..19] fp8: draft tiles
                       // landed / converted per producer warp, [20..21] fp8: tiles of parity 0 / 1 decoded (or
                       // passed through), a count that only grows
  int* len;
  int* base;
  int* lkind;          // fp8 cache: [kLandSlots] 1 when the slot's tile is a draft tile (nothing to decode)
};

__host__ __device__ inline size_t smem_bytes(int C, bool f8) {
  const int nk = f8 ? kF8NK : kNK, nv = f8 ? kF8NV : kNV;
  size_t off = static_cast<size_t>(nk + nv) * kKVBytes + kQBufBytes + (f8 ? kLandSlots * kLandBytes : 0);
  off += sizeof(uint64_t) * (2 * nk + 2 * nv + 2 + 3 * kNS + 3 + 2 * kLandSlots + 3);
  off += sizeof(uint64_t) * kMaxTreeNodes + sizeof(int) * kMaxTreeNodes;
  off += sizeof(float) * 2 * kQRows;
  off += sizeof(uint32_t) * 4 + sizeof(int) * kMiscInts;
  off += sizeof(int) * (2 * C + 1) + sizeof(int) * kLandSlots;
  return off + 1024;
}

__device__ Smem carve(uint8_t* raw, int C, bool f8) {
  const int nk = f8 ? kF8NK : kNK, nv = f8 ? kF8NV : kNV;
  Smem s;
  uint8_t* p = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  s.kring = p;
  p += nk * kKVBytes;
  s.vring = p;
  p += nv * kKVBytes;
  s.qbuf = p;
  p += kQBufBytes;
  s.land = p;
  if (f8) p += kLandSlots * kLandBytes;
  uint64_t* b = reinterpret_cast<uint64_t*>(p);
  s.kfull = b;
  s.kempty = s.kfull + nk;
  s.vfull = s.kempty + nk;
  s.vempty = s.vfull + nv;
  s.qfull = s.vempty + nv;
  s.qempty = s.qfull + 1;
  s.sfull = s.qempty + 1;
  s.sfree = s.sfull + kNS;
  s.pfull = s.sfree + kNS;
  s.ofree = s.pfull + kNS;
  s.mmadone = s.ofree + 1;
  s.lfull = s.mmadone + 2;
  s.lfree = s.lfull + kLandSlots;
  s.qland = s.lfree + kLandSlots;
  s.dland = s.qland + 1;
  s.anc = s.dland + 2;
  s.par = reinterpret_cast<int*>(s.anc + kMaxTreeNodes);
  s.comb = reinterpret_cast<float*>(s.par + kMaxTreeNodes);
  s.tmem_base = reinterpret_cast<uint32_t*>(s.comb + 2 * kQRows);
  s.misc = reinterpret_cast<int*>(s.tmem_base + 4);
  s.len = s.misc + kMiscInts;
  s.base = s.len + C;
  s.lkind = s.base + C + 1;
  return s;
}

// ------------------------------------------------------------ MMA issuer

// Two threads issue the MMAs, one stream each, so that neither stream's
// issue (which stalls while the tensor pipe is busy) delays the other:
// QK^T in tile order from warp kMmaWarp, P.V in tile order from warp
// kMmaPvWarp.  A tcgen05.commit tracks the MMAs of the thread that issues it.

// S = Q K^T of every tile.  Tile t needs its K tile, its S buffer freed by
// the completion of P.V of tile t - kNS, and (first tile of a piece) the
// piece's q block.
template <bool kF8>
__device__ __forceinline__ void run_mma_qk(const AttnParams& p, const Smem& sm, const Pipe& pipe, uint32_t tmem,
                                           Cursor cu) {
  // fp8 cache: q and the tiles are f16 (e4m3 -> f16 is one conversion per two codes).
  constexpr uint32_t idesc = kF8 ? idesc_f16(128, 64, false) : idesc_bf16(128, 64, false);
  constexpr int NK = kF8 ? kF8NK : kNK;
  int piece = 0;
  for (int t = 0; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    bool ok = !*pipe.abort;
    if (ok && ti.first) ok = mbar_wait(smem_addr(sm.qfull), piece & 1, p.err, p.wait_ns);
    if (ok && t >= kNS) ok = mbar_wait(smem_addr(&sm.sfree[t % kNS]), ((t - kNS) / kNS) & 1, p.err, p.wait_ns);
    if (ok) ok = mbar_wait(smem_addr(&sm.kfull[t % NK]), (t / NK) & 1, p.err, p.wait_ns);
    if (!ok) {
      *pipe.abort = 1;
      break;
    }
    if (ti.first) sm.misc[4] = ++piece;
    sm.misc[2] = t + 1;
    tc_fence_after();
    const uint32_t qbase = smem_addr(sm.qbuf);
    const uint32_t kbase = smem_addr(sm.kring + static_cast<size_t>(t % NK) * kKVBytes);
    // K tile: 8-key groups (the MMA's N direction) kGroupBytes apart and the dims 64..127 half
    // kGroupHalfBytes on (grouped layout), or 1 KB and kHalfBytes (halves layout).
    const bool grouped = ti.draft || p.prefix_grouped;
    const uint32_t half_off = grouped ? kGroupHalfBytes : kHalfBytes, group_off = grouped ? kGroupBytes : 1024;
#pragma unroll
    for (int ks = 0; ks < kHeadDim / 16; ++ks) {
      const uint64_t a = smem_desc_sw128(qbase + (ks >> 2) * (kQRows * 128) + (ks & 3) * 32, 16, 1024);
      const uint64_t b = smem_desc_sw128(kbase + (ks >> 2) * half_off + (ks & 3) * 32, 16, group_off);
      tc_mma(tmem + (t % kNS) * kTileKeys, a, b, idesc, ks > 0 ? 1u : 0u);
    }
    tc_commit(smem_addr(&sm.sfull[t % kNS]));
    tc_commit(smem_addr(&sm.kempty[t % NK]));
    if (ti.last) tc_commit(smem_addr(sm.qempty));
  }
  tc_commit(smem_addr(&sm.mmadone[0]));
}

// O_w += P V of every tile, w = t % 2 (the warpgroup that wrote P), with P
// read from tensor memory (the tile's S columns).  Tile t needs its P and its
// V tile; the first P.V into O_w of a piece (which overwrites O_w) needs the
// previous piece's epilogue to have read O.  Each completion frees the tile's
// S buffer for QK^T of tile t + kNS and tells the softmax that O_w holds P.V
// of tile t.
template <bool kF8>
__device__ __forceinline__ void run_mma_pv(const AttnParams& p, const Smem& sm, const Pipe& pipe, uint32_t tmem,
                                           Cursor cu) {
  constexpr uint32_t idesc = kF8 ? idesc_f16(128, 128, true) : idesc_bf16(128, 128, true);
  constexpr int NV = kF8 ? kF8NV : kNV;
  int piece = 0, piece_t0 = 0;
  for (int t = 0; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    if (ti.first) {
      ++piece;
      piece_t0 = t;
    }
    const bool first = t - piece_t0 < 2;
    bool ok = !*pipe.abort;
    if (ok && first && piece > 1) ok = mbar_wait(smem_addr(sm.ofree), (piece - 2) & 1, p.err, p.wait_ns);
    if (ok) ok = mbar_wait(smem_addr(&sm.pfull[t % kNS]), (t / kNS) & 1, p.err, p.wait_ns);
    if (ok) ok = mbar_wait(smem_addr(&sm.vfull[t % NV]), (t / NV) & 1, p.err, p.wait_ns);
    if (!ok) {
      *pipe.abort = 1;
      break;
    }
    sm.misc[6] = t + 1;
    tc_fence_after();
    const uint32_t pcol = tmem + (t % kNS) * kTileKeys;  // P: 32 columns of bf16 pairs
    const uint32_t vbase = smem_addr(sm.vring + static_cast<size_t>(t % NV) * kKVBytes);
    const uint32_t o = tmem + kTmemO + 128 * (t & 1);
    const bool grouped = ti.draft || p.prefix_grouped;
    const uint32_t half_off = grouped ? kGroupHalfBytes : kHalfBytes, group_off = grouped ? kGroupBytes : 1024;
#pragma unroll
    for (int k16 = 0; k16 < kTileKeys / 16; ++k16) {  // 16-key steps of the tile
      // V tile is MN-major: 64-dim halves `half_off` apart (leading), 8-key groups `group_off` apart (stride).
      const uint64_t bd = smem_desc_sw128(vbase + k16 * 2 * group_off, half_off, group_off);
      tc_mma_tmem_a(o, pcol + 8 * k16, bd, idesc, (first && k16 == 0) ? 0u : 1u);
    }
    tc_commit(smem_addr(&sm.vempty[t % NV]));
    tc_commit(smem_addr(&sm.sfree[t % kNS]));
  }
  tc_commit(smem_addr(&sm.mmadone[1]));
}

// e4m3 codes of one landed tile ([64 rows][128 codes] of K, then of V, 128-byte swizzle) -> f16 K and
// V tiles in the grouped layout, one hardware conversion per two codes (exact: 3 mantissa bits,
// exponents within f16's normal range); the power-of-two scales are applied by the consumers.  The
// four warps of a warpgroup share a tile: warp w decodes key rows 16 w .. 16 w + 15 (8-row groups
// 2 w, 2 w + 1) of K and of V.  Lane l takes 16-byte chunk c = l & 7 (dims 16c..16c+15) of rows
// 16 w + 4 i + (l >> 3), i = 0..3: rows 8k + r0 (even i) and 8k + 4 + r0 (odd i) take fixed
// swizzles, so every address is one of four per-lane bases plus a constant.  All eight loads of a
// lane go out before any conversion or store, so that their latencies overlap (K then V quarters one
// after the other measured 1% slower on the hybrid tree).
__device__ __forceinline__ void decode_e4m3_quarter_kv(uint32_t src, uint32_t dk, uint32_t dv, int lane, int w) {
  const uint32_t c = lane & 7, r0 = lane >> 3;
  const uint32_t s_even = src + r0 * 128 + ((c ^ r0) << 4);
  const uint32_t s_odd = src + (r0 + 4) * 128 + ((c ^ (r0 + 4)) << 4);
  const uint32_t dh = (c >> 2) * kGroupHalfBytes;
  const uint32_t e0 = dh + r0 * 128 + ((((2 * c) & 7) ^ r0) << 4);
  const uint32_t e1 = dh + r0 * 128 + ((((2 * c + 1) & 7) ^ r0) << 4);
  const uint32_t o0 = dh + (r0 + 4) * 128 + ((((2 * c) & 7) ^ (r0 + 4)) << 4);
  const uint32_t o1 = dh + (r0 + 4) * 128 + ((((2 * c + 1) & 7) ^ (r0 + 4)) << 4);
  const uint32_t k0 = 2 * static_cast<uint32_t>(w);
  uint4 v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
    v[i] = lds128((i & 1 ? s_odd : s_even) + (k0 + ((i >> 1) & 1)) * 1024 + (i >> 2) * (kLandBytes / 2));
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t k = k0 + ((i >> 1) & 1);
    const uint32_t dst = i < 4 ? dk : dv;
    const uint32_t ws[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
    uint32_t o[8];
#pragma unroll
    for (int q = 0; q < 4; ++q)
      asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %2;\n\t"
          "cvt.rn.f16x2.e4m3x2 %0, lo;\n\tcvt.rn.f16x2.e4m3x2 %1, hi;\n\t}"
          : "=r"(o[2 * q]), "=r"(o[2 * q + 1])
          : "r"(ws[q]));
    sts128(dst + (i & 1 ? o0 : e0) + k * kGroupBytes, make_uint4(o[0], o[1], o[2], o[3]));
    sts128(dst + (i & 1 ? o1 : e1) + k * kGroupBytes, make_uint4(o[4], o[5], o[6], o[7]));
  }
}

// ------------------------------------------------------------ softmax + epilogue

// Tile ownership: warpgroup w takes the tiles t with t % 2 == w (all 64 keys)
// with its own running max/sum and its own accumulator O_w in TMEM, so two
// tiles' softmax chains (S load, exponentials, P store) overlap; the two
// states are merged by log-sum-exp at the end of each piece.
// Row layout.  Dense units (more than 64 rows): thread = TMEM lane = stacked
// row 32 quarter + lane, holding all 64 S columns.  Spread units (at most 64
// rows): lanes 0..15 of each 32-lane quarter hold stacked rows 16 quarter +
// 0..15, so every SM sub-partition's softmax warps get rows; two threads share
// a lane (row), each with 32 of the 64 columns, and agree on the row max by
// one shuffle.
// O_wg *= alpha (per row) in TMEM, after P.V of this warpgroup's previous tile (t - 2) completed:
// sfree of its S buffer, which P.V commits when it completes.  A rescale needs an earlier tile of the
// piece, so t >= 2, and the wait is unambiguous: S of tile t implies that P.V of tile t - 4 (and
// so of t - 6) completed, and P.V of tile t + 2 cannot complete before this warpgroup's pfull of it.
template <bool kSpread>
__device__ __forceinline__ void rescale_o_tmem(const Smem& sm, const Pipe& pipe, const AttnParams& p, uint32_t my_o,
                                               int t, float alpha) {
  constexpr int kOChunks = kSpread ? 2 : 4;  // 32-column O chunks per thread
  if (!mbar_wait(smem_addr(&sm.sfree[(t - 2) % kNS]), ((t - 2) / kNS) & 1, p.err, p.wait_ns)) *pipe.abort = 1;
  tc_fence_after();
#pragma unroll
  for (int c = 0; c < kOChunks; ++c) {
    uint32_t o[32];
    if constexpr (kSpread) tmem_ld16x2_32(my_o + 32 * c, o);
    else tmem_ld32(my_o + 32 * c, o);
    tmem_wait_ld();
#pragma unroll
    for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * alpha);
    if constexpr (kSpread) tmem_st16x2_32(my_o + 32 * c, o);
    else tmem_st32(my_o + 32 * c, o);
  }
  tmem_wait_st();
}

template <bool kSpread, bool kF8>
__device__ __forceinline__ void run_softmax(const AttnParams& p, const Smem& sm, const Pipe& pipe, uint32_t tmem,
                                            Cursor cu) {
  constexpr int NK = kF8 ? kF8NK : kNK, NV = kF8 ? kF8NV : kNV;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3;                 // TMEM lanes this warp may access
  const int wg = warp >> 2;                     // warpgroup: owns tiles t with t % 2 == wg
  const int wtid = threadIdx.x & 127;           // thread within the warpgroup
  const int half = kSpread ? lane >> 4 : 0;     // spread: which 32 of the 64 columns
  const int tl = quarter * 32 + (kSpread ? (lane & 15) : lane);  // TMEM lane = row of the P buffer
  const int r = kSpread ? quarter * 16 + (lane & 15) : tl;       // stacked row of the unit
  constexpr int kCols = kSpread ? 32 : 64;      // S columns per thread
  constexpr int kOChunks = kSpread ? 2 : 4;     // 32-column O chunks per thread
  const int col0 = kCols * half;                // first S column of this thread
  const int warp_row0 = kSpread ? quarter * 16 : quarter * 32;
  const int tid = threadIdx.x;                  // 0..255 among the softmax threads
  const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
  const uint32_t my_o = trow + kTmemO + 128 * wg;
  const int HR = p.hkv * p.row_blocks;
  // Kernel parameters used per element, read once.
  const float qscale = p.qscale;
  const bool tree = p.tree != 0;
  const int nq = p.Nq, n_nodes = p.N;
  // Row bookkeeping of the current unit, recomputed when the unit changes.
  int unit_c = -1, unit_hr = -1, h = 0, rr = 0, nl = 0;
  bool valid = false, warp_live = false;
  float m_run = -INFINITY, l_run = 0.f;  // l_run: this thread's columns only (spread)
  int t = 0, anc_seq = -1;
  // fp8 cache: decodes tile y (its codes landed in slot y % kLandSlots) into its K and V ring slots with
  // this warpgroup's 128 threads, or passes a draft tile's landing through (its producer warp filled
  // the rings).  Tile y is decoded by warpgroup (y + 1) % 2 once it is done with tile y - kDecodeAhead
  // (its own tile; tiles 0..2 before the loop), so QK^T of tile y never waits for the warpgroup that
  // will take its softmax.  The ring-slot waits are unambiguous: that warpgroup has seen S of tile
  // y - 3, so QK^T of tile y - 2 NK and P.V of tile y - 2 NV had completed.
  const int ntiles = cu.t_end - cu.t_begin;
  auto decode_landed = [&](int y) {
    const int ls = y % kLandSlots;
    bool good = !*pipe.abort && mbar_wait(smem_addr(&sm.lfull[ls]), (y / kLandSlots) & 1, p.err, p.wait_ns);
    const bool landed = good;
    const bool codes = good && sm.lkind[ls] == 0;
    if (codes) {
      good = mbar_wait(smem_addr(&sm.kempty[y % NK]), ((y / NK) & 1) ^ 1u, p.err, p.wait_ns) &&
             mbar_wait(smem_addr(&sm.vempty[y % NV]), ((y / NV) & 1) ^ 1u, p.err, p.wait_ns);
      if (good) {
        const uint32_t src = smem_addr(sm.land + static_cast<size_t>(ls) * kLandBytes);
        decode_e4m3_quarter_kv(src, smem_addr(sm.kring + static_cast<size_t>(y % NK) * kKVBytes),
                               smem_addr(sm.vring + static_cast<size_t>(y % NV) * kKVBytes), lane, quarter);
        fence_proxy_async_smem();  // the MMAs read the tiles through the async proxy
      }
    }
    if (!good) *pipe.abort = 1;
    named_barrier_sync(kBarDecode0 + wg, kSoftmaxThreads / 2);
    if (wtid == 0) {
      if (codes && good) {
        mbar_arrive(smem_addr(&sm.kfull[y % NK]));
        mbar_arrive(smem_addr(&sm.vfull[y % NV]));
      }
      if (landed) {
        mbar_arrive(smem_addr(&sm.lfree[ls]));
        sm.misc[14 + (y & 1)] = (y >> 1) + 1;
      }
      reinterpret_cast<volatile int*>(sm.misc)[20 + (y & 1)] = (y >> 1) + 1;  // tile y decoded
    }
  };
  // Outputs and the workspace are written only once the preceding kernel has ended
  // (KVSHOT_OVERLAP_PREVIOUS); the first S needs q, which comes after that anyway.
  wait_for_prerequisite_grid();
  if constexpr (kF8) {
    for (int y = 1 - wg; y < min(kDecodeAhead, ntiles); y += 2) decode_landed(y);
  }
  for (; cu.t < cu.t_end; cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    if (cu.c != unit_c || cu.hr != unit_hr) {
      unit_c = cu.c;
      unit_hr = cu.hr;
      h = cu.hr / p.row_blocks;
      const int rb = cu.hr - h * p.row_blocks;
      const int rows_blk = min(p.rows_per_unit, p.rows_total - rb * p.rows_per_unit);
      valid = r < rows_blk;
      warp_live = warp_row0 < rows_blk;
      rr = rb * p.rows_per_unit + r;
      nl = valid ? rr / p.G : 0;
    }
    if (ti.first) {
      m_run = -INFINITY;
      l_run = 0.f;
    }
    if (ti.draft && tree) {
      const int seq = cu.c / (p.C / p.B);
      if (seq != anc_seq) {
        build_ancestor_masks(p, seq, sm.anc, sm.par, tid, kSoftmaxThreads, kBarSoftmax);
        anc_seq = seq;
      }
    }
    bool live = !*pipe.abort;
    if ((t & 1) == wg) {
      const int sbuf = t % kNS;
      if (live && !mbar_wait(smem_addr(&sm.sfull[sbuf]), (t / kNS) & 1, p.err, p.wait_ns)) {
        *pipe.abort = 1;
        live = false;
      }
      live = __all_sync(0xffffffffu, live);
      tc_fence_after();
      float pr[kCols];
      bool any_rescale = false;  // dense rows: some row of this warp moves its reference max, O_wg is rescaled
      float alpha = 1.f;         // dense rows: this row's factor
      if (live && warp_live) {
        uint32_t sv[kCols];
        if constexpr (kSpread) {
          tmem_ld16x2_32_s32(trow + sbuf * kTileKeys, sv);
        } else {
          tmem_ld32(trow + sbuf * kTileKeys, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
          tmem_ld32(trow + sbuf * kTileKeys + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
        }
        tmem_wait_ld();
        // Visible keys of this row (bit j = key key0 + j).
        uint64_t v64 = 0;
        if (valid) {
          v64 = ti.nkeys >= 64 ? ~0ull : ((1ull << ti.nkeys) - 1ull);
          if (ti.draft) {
            uint64_t dm;
            if (tree) {
              dm = sm.anc[min(nl, nq - 1)] >> ti.key0;  // tree drafts have N <= 64, so key0 == 0
            } else {
              const int last = n_nodes - nq + nl - ti.key0;  // chain: slots key0 .. node are visible
              dm = last >= 63 ? ~0ull : (last < 0 ? 0ull : ((2ull << last) - 1ull));
            }
            v64 &= dm;
          }
        }
        const uint64_t vis = v64 >> col0;  // bit j = column col0 + j
        // fp8 cache: the prefix keys' power-of-two scale is part of the score scale.
        const float qs = (kF8 && !ti.draft) ? qscale * p.k_scale : qscale;
        float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        // Spread rows keep the raw scores and fold the scale into the exponent's argument,
        // 2^(s qs - m) = ex2(fma(s, qs, -m)), with the row max taken on the raw scores (qs > 0), in
        // two-lane FMAs and adds and three-input maxima (row_max, row_exp): fewer instructions per
        // score (per-depth hybrid tree 55.0 -> 53.7 us per call on GB300 for the folded scale alone).
        // Dense rows measured 2% slower with the folded scale and scale each score first.
        const float pre = kSpread ? 1.f : qs;  // spread rows: pr holds the raw scores
        // Dense rows skip the per-key mask on a full prefix tile (every key is visible): +6% on the
        // 128-row whole-tree stacks; spread rows (half the columns) measured ~2-4% slower with it.
        if (!kSpread && valid && !ti.draft && ti.nkeys >= kTileKeys) {
#pragma unroll
          for (int j = 0; j < kCols; ++j) {
            pr[j] = __uint_as_float(sv[j]) * pre;
            mx4[j & 3] = fmaxf(mx4[j & 3], pr[j]);
          }
        } else {
#pragma unroll
          for (int j = 0; j < kCols; ++j) {
            pr[j] = ((vis >> j) & 1u) ? __uint_as_float(sv[j]) * pre : -INFINITY;
            if constexpr (!kSpread) mx4[j & 3] = fmaxf(mx4[j & 3], pr[j]);
          }
        }
        float mx;
        if constexpr (kSpread) mx = row_max(pr) * qs;
        else mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
        if constexpr (kSpread) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        // Lazy rescale: move this row's reference max only when it grows by > 2^8.  Dense rows rescale
        // O_wg after P is stored (below), so that P's 64 registers are free by then (it removed the
        // dense variant's spills); spread rows, with half the columns, rescale here, which measured
        // faster for them.
        const bool grow = valid && (m_run == -INFINITY ? mx != -INFINITY : mx > m_run + kRescaleThreshold);
        const bool rescale_o = grow && m_run != -INFINITY;
        if constexpr (kSpread) {
          if (__any_sync(0xffffffffu, rescale_o)) {
            const float a = rescale_o ? ex2(m_run - mx) : 1.f;
            rescale_o_tmem<kSpread>(sm, pipe, p, my_o, t, a);
            l_run *= a;
          }
        } else {
          any_rescale = __any_sync(0xffffffffu, rescale_o);
          alpha = rescale_o ? ex2(m_run - mx) : 1.f;
          l_run *= alpha;
        }
        if (grow) m_run = mx;
        const float m_use = m_run == -INFINITY ? 0.f : m_run;
        uint32_t pk[kCols / 2];  // P as bf16 pairs over the S columns just read (rows past the stack: zeros)
        // fp8 cache: P of prefix tiles carries the values' power-of-two scale; the running sum does not.
        const float vs = (kF8 && !ti.draft) ? p.v_scale : 1.f;
        if constexpr (kSpread) {
          l_run += row_exp<kCols, kF8>(pr, qs, m_use, vs, pk);
        } else {
          float ps4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int j = 0; j < kCols / 2; ++j) {
            const float e0 = ex2(pr[2 * j] - m_use), e1 = ex2(pr[2 * j + 1] - m_use);
            ps4[(2 * j) & 3] += e0;
            ps4[(2 * j + 1) & 3] += e1;
            pk[j] = kF8 ? pack_f16x2_tc(e0 * vs, e1 * vs) : pack_bf16x2(e0 * vs, e1 * vs);
          }
          l_run += (ps4[0] + ps4[1]) + (ps4[2] + ps4[3]);
        }
        if constexpr (kSpread) tmem_st16x2_16(trow + sbuf * kTileKeys, pk);
        else tmem_st32(trow + sbuf * kTileKeys, pk);
      }
      // Spread rows release P of this tile without waiting for P.V of this warpgroup's previous tile;
      // only a rescale of O_wg waits for it (rescale_o_tmem).  Dense rows wait for it on every tile:
      // releasing P earlier measured slower for them (whole-tree multi-layer tree 377 -> 384 us per
      // call on GB300), while the spread rows gained 0.3-1%.
      if constexpr (!kSpread) {
        if (live && t >= 2 && !mbar_wait(smem_addr(&sm.sfree[(t - 2) % kNS]), ((t - 2) / kNS) & 1, p.err, p.wait_ns))
          *pipe.abort = 1;
        if (live && warp_live && any_rescale) rescale_o_tmem<kSpread>(sm, pipe, p, my_o, t, alpha);
      }
      if (live && warp_live) tmem_wait_st();
      if (live && ti.nkeys < kTileKeys) {
        // V rows past the valid keys may hold NaN; 0 * NaN would poison P.V.
        if (!mbar_wait(smem_addr(&sm.vfull[t % NV]), (t / NV) & 1, p.err, p.wait_ns)) *pipe.abort = 1;
        uint8_t* vptr = sm.vring + static_cast<size_t>(t % NV) * kKVBytes;
        const int nz = (kTileKeys - ti.nkeys) * 16;
        for (int i = wtid; i < nz; i += kSoftmaxThreads / 2) {
          const int key = ti.nkeys + (i >> 4), ch = i & 15;
          *reinterpret_cast<uint4*>(vptr + tile_off_tc(key, ch, ti.draft || p.prefix_grouped)) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();  // the zeros, written through the generic proxy, are read by P.V
      }
      tc_fence_before();
      mbar_arrive(smem_addr(&sm.pfull[sbuf]));
      if constexpr (kF8) {
        if (t + kDecodeAhead < ntiles) decode_landed(t + kDecodeAhead);
      }
    }
    if (ti.last) {
      // Every P.V of the piece has completed once P.V of tile t has (P.V
      // completes in tile order; sfree of the tile's S buffer).  The owner of
      // tile t saw S of it, so P.V of tile t - 4 had completed and the wait is
      // unambiguous; the other warpgroup saw S of tile t - 1 only, so it first
      // waits P.V of its own tile t - 1 (after which P.V of t - 4 has completed).
      bool ok = live;
      if (ok && (t & 1) != wg && t >= 1)
        ok = mbar_wait(smem_addr(&sm.sfree[(t - 1) % kNS]), ((t - 1) / kNS) & 1, p.err, p.wait_ns);
      ok = ok && mbar_wait(smem_addr(&sm.sfree[t % kNS]), (t / kNS) & 1, p.err, p.wait_ns);
      ok = __all_sync(0xffffffffu, ok);
      tc_fence_after();
      float l_row = l_run;
      if constexpr (kSpread) l_row += __shfl_xor_sync(0xffffffffu, l_run, 16);
      // Merge the two warpgroups' states: warpgroup 1 publishes (max, sum), warpgroup 0 writes the row.
      if (wg == 1) {
        sm.comb[2 * tl] = m_run;
        sm.comb[2 * tl + 1] = l_row;
      }
      named_barrier_sync(kBarSoftmax, kSoftmaxThreads);
      tc_fence_after();
      if (wg == 0 && ok && warp_live) {
        const float m1 = sm.comb[2 * tl], l1 = sm.comb[2 * tl + 1];
        const float M = fmaxf(m_run, m1);
        const float w0 = m_run == -INFINITY ? 0.f : ex2(m_run - M);
        const float w1 = m1 == -INFINITY ? 0.f : ex2(m1 - M);
        const float L = w0 * l_row + w1 * l1;
        const float inv = L > 0.f ? 1.f / L : 0.f;
        // A warpgroup that owned no tile of this piece left O_w untouched: its weight is 0 and O_w is skipped.
        const float a0 = w0 * inv, a1 = w1 * inv;
        const float lse2 = L > 0.f ? M + __log2f(L) : -INFINITY;
        const bool whole = cu.lt == cu.ut - 1 && (cu.t - cu.t_begin) >= cu.lt;
        const int slot = cu.c * HR + cu.hr + blockIdx.x;
        size_t orow = 0;
        if (valid && whole) {
          const int g = rr - nl * p.G;
          orow = (static_cast<size_t>(cu.c) * p.Nq + nl) * p.hq + h * p.G + g;
        }
#pragma unroll 1
        for (int c = 0; c < kOChunks; ++c) {
          uint32_t o0[32], o1[32];
          if constexpr (kSpread) {
            tmem_ld16x2_32(trow + kTmemO + 32 * c, o0);
            tmem_ld16x2_32(trow + kTmemO + 128 + 32 * c, o1);
          } else {
            tmem_ld32(trow + kTmemO + 32 * c, o0);
            tmem_ld32(trow + kTmemO + 128 + 32 * c, o1);
          }
          tmem_wait_ld();
          const int d0 = kSpread ? 64 * half + 32 * c : 32 * c;  // first output dim of this chunk
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j)
            v[j] = (a0 != 0.f ? a0 * __uint_as_float(o0[j]) : 0.f) + (a1 != 0.f ? a1 * __uint_as_float(o1[j]) : 0.f);
          if (valid) {
            if (whole) {
              uint4* dst = reinterpret_cast<uint4*>(p.out + orow * kHeadDim + d0);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                uint4 w;
                w.x = pack_bf16x2(v[8 * k + 0], v[8 * k + 1]);
                w.y = pack_bf16x2(v[8 * k + 2], v[8 * k + 3]);
                w.z = pack_bf16x2(v[8 * k + 4], v[8 * k + 5]);
                w.w = pack_bf16x2(v[8 * k + 6], v[8 * k + 7]);
                dst[k] = w;
              }
            } else {
              float4* dst = reinterpret_cast<float4*>(
                  p.ws_o + (static_cast<size_t>(slot) * p.rows_per_unit + r) * kHeadDim + d0);
#pragma unroll
              for (int k = 0; k < 8; ++k) dst[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
            }
          }
        }
        if (valid && half == 0) {
          if (whole) p.lse[orow] = lse2 * 0.69314718055994531f;
          else p.ws_lse[static_cast<size_t>(slot) * p.rows_per_unit + r] = lse2;
        }
      }
      named_barrier_sync(kBarSoftmax, kSoftmaxThreads);  // comb is reused at the next piece end
      tc_fence_before();
      mbar_arrive(smem_addr(sm.ofree));
    }
    ++t;
  }
}

// ------------------------------------------------------------ TMA producer

// Exact n / d for 0 <= n < 2^24 and 1 <= d <= 256 by a multiply-high with
// m = ceil(2^32 / d): writing n = q d + r, the product overshoots n / d by
// n (m d - 2^32) / (d 2^32) < 1 / d, which never carries r / d past 1.
// Larger dividends (`small` false) take the hardware division.
struct FastDiv {
  uint32_t d, m;
  bool exact;
  __device__ __forceinline__ FastDiv(uint32_t dd, bool small)
      : d(dd), m(dd > 1 ? 0xFFFFFFFFu / dd + 1u : 0u), exact(small && dd <= 256) {}
  __device__ __forceinline__ int div(int n) const {
    const uint32_t u = static_cast<uint32_t>(n);
    return static_cast<int>(d == 1 ? u : (exact ? __umulhi(u, m) : u / d));
  }
};

// TMA boxes of one K (or V) tile; this lane's box is i = lane & 15 (at most
// 8 per tensor).  Grouped layout (draft tiles, and prefix tiles when
// p.prefix_grouped): a box holds whole 8-key groups with both 64-dim halves
// (a page of P <= 64 tokens, a 64-token slice of a larger page or of the
// contiguous cache, or 8 draft slots); halves layout (a contiguous cache whose
// l_cap is not a multiple of 8): one box per 64-dim half.  h is the unit's KV
// head, `pages` the cache's pages in use.  Warp-wide.
struct TileBoxes {
  bool draft, grouped;
  int nbox;        // boxes per tensor
  int x, y;        // this lane's box: map coordinates (x: halves layout only)
  uint32_t off;    // this lane's box: byte offset in the tile
  uint32_t bytes;  // bytes of all of one tensor's boxes
};

__device__ __forceinline__ TileBoxes tile_boxes(const AttnParams& p, const Cursor& cu, PageWindow& win, int lane,
                                                int h, int pages, const FastDiv& pdiv) {
  TileBoxes tb;
  tb.draft = cu.lt >= cu.pt;
  tb.grouped = tb.draft || p.prefix_grouped;
  tb.x = 0;
  const int key0 = (tb.draft ? cu.lt - cu.pt : cu.lt) * kTileKeys;
  const int nkeys = min(kTileKeys, (tb.draft ? p.N : cu.L) - key0);
  const int i = lane & 15;
  if (tb.draft) {
    // 3-D map {64 dims, rows, 2 halves}: first row of the box.
    tb.nbox = (nkeys + kDraftBoxRows - 1) / kDraftBoxRows;
    tb.y = (cu.c * p.hkv + h) * p.n_max + key0 + i * kDraftBoxRows;
    tb.off = static_cast<uint32_t>(i) * kGroupBytes;
    tb.bytes = static_cast<uint32_t>(tb.nbox) * kGroupBytes;
  } else if (p.paged) {
    // 4-D map {64 dims, 8 rows, 2 halves, row groups}: row group of the box.  Pages of
    // P <= 64 tokens: one box per page (P divides the tile); larger pages: one 64-row box.
    const int P = p.page_size;
    const bool small_pages = P < kTileKeys;
    tb.nbox = small_pages ? pdiv.div(nkeys + P - 1) : 1;
    const int pg0 = pdiv.div(key0);
    const int npg = small_pages ? tb.nbox : 1;
    win.cover(p, cu.c, pages, pg0, npg, lane);
    const int pid = win.get(pg0 + (small_pages ? min(i, npg - 1) : 0));
    tb.y = ((pid * p.hkv + h) * P + (small_pages ? 0 : key0 - pg0 * P)) >> 3;
    const uint32_t box_bytes = small_pages ? static_cast<uint32_t>(P) * 256u : kKVTileBytes;
    tb.off = static_cast<uint32_t>(i) * box_bytes;
    tb.bytes = static_cast<uint32_t>(tb.nbox) * box_bytes;
  } else if (p.prefix_grouped) {
    tb.nbox = 1;
    tb.y = ((cu.c * p.hkv + h) * p.l_cap + key0) >> 3;
    tb.off = 0;
    tb.bytes = kKVTileBytes;
  } else {
    // 2-D map {128 dims, rows}, boxes {64 dims, 64 rows}: box i is half i.
    tb.nbox = 2;
    tb.x = i * 64;
    tb.y = (cu.c * p.hkv + h) * p.l_cap + key0;
    tb.off = static_cast<uint32_t>(i) * kHalfBytes;
    tb.bytes = kKVTileBytes;
  }
  return tb;
}

// Walks this CTA's tiles and loads those with t % 2 == role: their K tile
// into the K ring and their V tile into the V ring, each box from its own
// lane.  Two producer warps keep twice the loads in flight that one warp can
// (a warp's bulk-tensor issues stall while its earlier ones are outstanding),
// and each tile's page lookups are done once for both rings.
// The q block of every piece (single buffer) is loaded by role 1 alone (so the
// first tile's K and V, from role 0, do not queue behind it): an
// mbarrier wait by parity cannot tell a phase from the one two phases
// earlier, so the q-buffer release must be waited by a thread that also
// waited its previous phase.  (A ring slot is safe to wait from either warp:
// its release is an in-order MMA completion that the warp's own previous
// wait already covers two phases back.)  A spread unit's q block goes in
// boxes of 16 stacked rows, box k to TMEM lanes (= q buffer rows)
// 32 k .. 32 k + 15.  misc[8 + role] / misc[10 + role]: one past the last K /
// V tile this warp issued (read by the drain after an abort).
template <int kMode, class SM>
__device__ __forceinline__ void run_producer_tc(const AttnParams& p, const TensorMaps& maps, const SM& sm,
                                                const Pipe& pipe, Cursor cu, int nq_box, int role) {
  constexpr bool kSpread = kMode == kModeSpread;
  constexpr int NK = RingOf<kMode>::NK, NV = RingOf<kMode>::NV;
  const int lane = threadIdx.x & 31;
  const uint64_t policy = l2_policy_evict_first();
  PageWindow win;
  int t = 0, piece = 0;
  const int rows_q = p.G * nq_box;
  const bool small = p.len_bound < (1 << 24) - 2 * kTileKeys;
  const FastDiv pdiv(p.paged ? p.page_size : 1, small), rbdiv(p.row_blocks, true);
  int unit_c = -1, unit_hr = -1, h = 0, pages = 0;  // the current unit's KV head and its cache's pages
  int ok = 1;
  bool waited = false;  // griddepcontrol.wait done
  for (; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const bool first = cu.t == cu.t_begin || cu.lt == 0;  // first tile of a piece
    const bool mine = (t & 1) == role;
    if (!mine && !(first && role == 1)) {
      piece += first;
      continue;
    }
    if (cu.c != unit_c || cu.hr != unit_hr) {
      unit_c = cu.c;
      unit_hr = cu.hr;
      h = rbdiv.div(cu.hr);
      pages = p.paged ? pdiv.div(cu.L + p.page_size - 1) : 0;
    }
    if (first && role == 1) {  // the unit's q block
      if (!waited) {  // q may come from the preceding kernel (KVSHOT_OVERLAP_PREVIOUS)
        wait_for_prerequisite_grid();
        waited = true;
      }
      if (lane == 0) {
        const uint32_t qbar = smem_addr(sm.qfull);
        ok = mbar_wait(smem_addr(sm.qempty), (piece & 1) ^ 1u, p.err, p.wait_ns) && !*pipe.abort;
        if (ok) {
          const int rb = cu.hr - h * p.row_blocks;
          const uint32_t dst = smem_addr(sm.qbuf);
          if constexpr (kMode == kModePair) {
            // Q_0 and Q_1: the unit's two blocks of nq_box draft nodes x G heads (128 rows each).
            mbar_arrive_expect_tx(qbar, 4 * kQRows * 128);
            for (int w = 0; w < 2; ++w) {
              const uint32_t d = dst + w * kQBufBytes;
              const int node0 = (2 * rb + w) * nq_box;
              tma_load_4d(d, &maps.q, 0, h * p.G, node0, cu.c, qbar);
              tma_load_4d(d + kQRows * 128, &maps.q, 64, h * p.G, node0, cu.c, qbar);
            }
          } else {
            const QBox qb = q_box(p.G, nq_box, kSpread);
            const int box_rows = qb.heads * qb.nodes;
            const int nqb = kSpread ? (rows_q + box_rows - 1) / box_rows : 1;
            mbar_arrive_expect_tx(qbar, 2 * nqb * box_rows * 128);
            for (int k = 0; k < nqb; ++k) {
              const int s0 = k * box_rows;  // first stacked row of the box
              const uint32_t d = dst + k * 32 * 128;
              tma_load_4d(d, &maps.q, 0, h * p.G + s0 % p.G, rb * nq_box + s0 / p.G, cu.c, qbar);
              tma_load_4d(d + kQRows * 128, &maps.q, 64, h * p.G + s0 % p.G, rb * nq_box + s0 / p.G, cu.c, qbar);
            }
          }
          sm.misc[3] = piece + 1;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) *pipe.abort = 1;
        break;
      }
    }
    piece += first;
    if (!mine) continue;
    const TileBoxes tb = tile_boxes(p, cu, win, lane, h, pages, pdiv);
    if (tb.draft && !waited) {  // so may the draft K/V; the target K/V before them may not
      wait_for_prerequisite_grid();
      waited = true;
    }
    // Lanes 0..15 load the K boxes, lanes 16..31 the V boxes (box = lane & 15).
    const int kv = lane >> 4, i = lane & 15;
    const int kslot = t % NK, vslot = t % NV;
    // A V slot is free once P.V of its previous tile completed, a K slot once QK^T of its previous tile
    // (t - NK) completed; each slot has its own release barrier, whose next completion (tile t) needs
    // this very load, so a phase is never mistaken for one two phases later.  Lane 0 waits for the K
    // slot and lane 1 for the V slot together.
    if (lane < 2 && ok) {
      const uint32_t bar = lane == 0 ? smem_addr(&sm.kempty[kslot]) : smem_addr(&sm.vempty[vslot]);
      const uint32_t par = ((t / (lane == 0 ? NK : NV)) & 1) ^ 1u;
      ok = mbar_wait(bar, par, p.err, p.wait_ns) && !*pipe.abort;
    }
    ok = __all_sync(0xffffffffu, ok);
    if (!ok) {
      if (lane == 0) *pipe.abort = 1;
      break;
    }
    const uint32_t full_bar = smem_addr(kv ? &sm.vfull[vslot] : &sm.kfull[kslot]);
    if ((lane & 15) == 0) mbar_arrive_expect_tx(full_bar, tb.bytes);
    if (i < tb.nbox) {
      const uint32_t dst = smem_addr((kv ? sm.vring + static_cast<size_t>(vslot) * kKVBytes
                                         : sm.kring + static_cast<size_t>(kslot) * kKVBytes)) +
                           tb.off;
      if (tb.draft) tma_load_3d(dst, kv ? &maps.dv : &maps.dk, 0, tb.y, 0, full_bar, policy);
      else if (tb.grouped) tma_load_4d_hint(dst, kv ? &maps.tv : &maps.tk, 0, 0, 0, tb.y, full_bar, policy);
      else tma_load_2d(dst, kv ? &maps.tv : &maps.tk, tb.x, tb.y, full_bar, policy);
    }
    if (lane == 0) {
      sm.misc[8 + role] = t + 1;
      sm.misc[10 + role] = t + 1;
    }
    if (!ok) {
      if (lane == 0) *pipe.abort = 1;
      break;
    }
  }
}



// ------------------------------------------------------------ fp8 target cache

// TMA boxes of the e4m3 codes of one prefix tile (2-D map {128 codes, rows}, boxes of whole 128-byte
// rows, 128-byte swizzle): pages of P < 64 tokens one box each, larger pages and the contiguous cache
// one 64-row box.  This lane's box is i = lane & 15; rows land in order at 128 bytes each.
__device__ __forceinline__ TileBoxes tile_boxes_f8(const AttnParams& p, const Cursor& cu, PageWindow& win, int lane,
                                                   int h, int pages, const FastDiv& pdiv) {
  TileBoxes tb;
  tb.draft = false;
  tb.grouped = true;
  tb.x = 0;
  const int key0 = cu.lt * kTileKeys;
  const int nkeys = min(kTileKeys, cu.L - key0);
  const int i = lane & 15;
  if (p.paged) {
    const int P = p.page_size;
    const bool small_pages = P < kTileKeys;
    const int br = small_pages ? P : kTileKeys;
    tb.nbox = small_pages ? pdiv.div(nkeys + P - 1) : 1;
    const int pg0 = pdiv.div(key0);
    win.cover(p, cu.c, pages, pg0, tb.nbox, lane);
    const int pid = win.get(pg0 + (small_pages ? min(i, tb.nbox - 1) : 0));
    tb.y = (pid * p.hkv + h) * P + (small_pages ? 0 : key0 - pg0 * P);
    tb.off = static_cast<uint32_t>(i * br * 128);
    tb.bytes = static_cast<uint32_t>(tb.nbox * br * 128);
  } else {
    tb.nbox = 1;
    tb.y = (cu.c * p.hkv + h) * p.l_cap + key0;
    tb.off = 0;
    tb.bytes = kTileKeys * 128;
  }
  return tb;
}

// Producer warp `role` with an fp8 target cache; its tiles are t % 2 == role.  A prefix tile's e4m3
// codes land in landing slot t % kLandSlots once the decode of tile t - kLandSlots has freed it; the
// softmax warpgroups decode them into the f16 ring tiles (decode_landed in run_softmax), which keeps
// the decode (and its shared-memory traffic) off this warp, whose box issues and waits then bound
// nothing.  A draft tile (bf16) is loaded straight into its ring slots and converted to f16 in place
// here, and its landing slot is passed through (lkind 1) so that every tile takes one phase of its
// slot's barriers.  q blocks as in run_producer_tc (role 1), converted to f16 here.
__device__ __forceinline__ void run_producer_f8(const AttnParams& p, const TensorMaps& maps, const Smem& sm,
                                                const Pipe& pipe, Cursor cu, int nq_box, int role) {
  constexpr int NK = kF8NK, NV = kF8NV;
  const int lane = threadIdx.x & 31;
  const uint64_t policy = l2_policy_evict_first();
  PageWindow win;
  int t = 0, piece = 0;
  const bool small = p.len_bound < (1 << 24) - 2 * kTileKeys;
  const FastDiv pdiv(p.paged ? p.page_size : 1, small), rbdiv(p.row_blocks, true);
  int unit_c = -1, unit_hr = -1, h = 0, pages = 0;
  int ok = 1;
  bool waited = false;
  int drafts = 0, qblocks = 0, issued = 0;  // draft tiles loaded, q blocks converted, own tiles issued
  for (; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const bool first = cu.t == cu.t_begin || cu.lt == 0;  // first tile of a piece
    const bool mine = (t & 1) == role;
    if (!mine && !(first && role == 1)) {
      piece += first;
      continue;
    }
    if (cu.c != unit_c || cu.hr != unit_hr) {
      unit_c = cu.c;
      unit_hr = cu.hr;
      h = rbdiv.div(cu.hr);
      pages = p.paged ? pdiv.div(cu.L + p.page_size - 1) : 0;
    }
    if (first && role == 1) {  // the unit's q block (released by QK^T of the previous piece's last tile)
      if (!waited) {
        wait_for_prerequisite_grid();
        waited = true;
      }
      if (lane == 0) {
        const uint32_t qbar = smem_addr(sm.qland);  // converted to f16 below, then qfull
        ok = mbar_wait(smem_addr(sm.qempty), (piece & 1) ^ 1u, p.err, p.wait_ns) && !*pipe.abort;
        if (ok) {
          const int rb = cu.hr - h * p.row_blocks;
          const uint32_t dst = smem_addr(sm.qbuf);
          const QBox qb = q_box(p.G, nq_box, nq_box * p.G <= kSpreadMaxRows);
          const int box_rows = qb.heads * qb.nodes;
          const int rows_q = p.G * nq_box;
          const int nqb = nq_box * p.G <= kSpreadMaxRows ? (rows_q + box_rows - 1) / box_rows : 1;
          mbar_arrive_expect_tx(qbar, 2 * nqb * box_rows * 128);
          for (int k = 0; k < nqb; ++k) {
            const int s0 = k * box_rows;
            const uint32_t d = dst + k * 32 * 128;
            tma_load_4d(d, &maps.q, 0, h * p.G + s0 % p.G, rb * nq_box + s0 / p.G, cu.c, qbar);
            tma_load_4d(d + kQRows * 128, &maps.q, 64, h * p.G + s0 % p.G, rb * nq_box + s0 / p.G, cu.c, qbar);
          }
          sm.misc[3] = piece + 1;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(smem_addr(sm.qland), qblocks & 1, p.err, p.wait_ns));
      if (!ok) {
        if (lane == 0) *pipe.abort = 1;
        break;
      }
      ++qblocks;
      bf16_to_f16_inplace(smem_addr(sm.qbuf), kQBufBytes, lane);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_addr(sm.qfull));
        sm.misc[1] = qblocks;
      }
    }
    piece += first;
    if (!mine) continue;
    const bool draft = cu.lt >= cu.pt;
    const TileBoxes tb = draft ? tile_boxes(p, cu, win, lane, h, pages, pdiv) : tile_boxes_f8(p, cu, win, lane, h,
                                                                                                pages, pdiv);
    const int ls = t % kLandSlots;
    const uint32_t lbar = smem_addr(&sm.lfull[ls]);
    // The landing slot is free once tile t - kLandSlots (this warp's, two own tiles back) was decoded.
    // The wait is unambiguous because kLandSlots is even: the slot's previous release, the decode of
    // tile t - 2 kLandSlots, was waited by this warp before it landed tile t - kLandSlots.  (With an
    // odd count the slot alternates between the two warps and this wait could pass two phases early.)
    if (lane == 0)
      ok = mbar_wait(smem_addr(&sm.lfree[ls]), ((t / kLandSlots) & 1) ^ 1u, p.err, p.wait_ns) && !*pipe.abort;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) {
      if (lane == 0) *pipe.abort = 1;
      break;
    }
    const int kv = lane >> 4, i = lane & 15;
    if (draft) {
      const int kslot = t % NK, vslot = t % NV;
      int good = 1;
      // This warp waits for the ring slots only at its draft tiles, so by itself it cannot know that the
      // slots' earlier releases have happened (a wait by parity could then pass two phases early).  Tile
      // t - 1 being decoded means its decoder had seen S of tile t - 4: QK^T of tile t - 4 and P.V of
      // tile t - 8 had completed, which makes the waits below unambiguous.  A growing count, not a
      // barrier phase, so the poll cannot be ambiguous itself.
      if (t >= 1) {
        const int need = ((t - 1) >> 1) + 1;
        volatile int* dec = &sm.misc[20 + ((t - 1) & 1)];
        const uint64_t t0 = global_timer_ns();
        while (good && *dec < need) {
          if (*pipe.abort) good = 0;
          else if (global_timer_ns() - t0 > p.wait_ns) {
            set_error(p.err, KVSHOT_ERR_TIMEOUT);
            good = 0;
          }
        }
      }
      if (lane < 2 && good) {
        const uint32_t bar = lane == 0 ? smem_addr(&sm.kempty[kslot]) : smem_addr(&sm.vempty[vslot]);
        const uint32_t par = ((t / (lane == 0 ? NK : NV)) & 1) ^ 1u;
        good = mbar_wait(bar, par, p.err, p.wait_ns) && !*pipe.abort;
      }
      if (!__all_sync(0xffffffffu, good)) {
        ok = 0;
        if (lane == 0) *pipe.abort = 1;
        break;
      }
      if (!waited) {  // the draft K/V may come from the preceding kernel (KVSHOT_OVERLAP_PREVIOUS)
        wait_for_prerequisite_grid();
        waited = true;
      }
      // bf16 draft K/V land in the ring slots and are converted to f16 there.
      uint8_t* kd = sm.kring + static_cast<size_t>(kslot) * kKVBytes;
      uint8_t* vd = sm.vring + static_cast<size_t>(vslot) * kKVBytes;
      const uint32_t dbar = smem_addr(&sm.dland[role]);
      if (lane == 0) mbar_arrive_expect_tx(dbar, 2 * tb.bytes);
      __syncwarp();
      if (i < tb.nbox) tma_load_3d(smem_addr(kv ? vd : kd) + tb.off, kv ? &maps.dv : &maps.dk, 0, tb.y, 0, dbar,
                                   policy);
      if (lane == 0) sm.misc[16 + role] = drafts + 1;
      if (!__all_sync(0xffffffffu, mbar_wait(dbar, drafts & 1, p.err, p.wait_ns))) {
        ok = 0;
        if (lane == 0) *pipe.abort = 1;
        break;
      }
      ++drafts;
      bf16_to_f16_inplace(smem_addr(kd), kKVBytes, lane);
      bf16_to_f16_inplace(smem_addr(vd), kKVBytes, lane);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_addr(&sm.kfull[kslot]));
        mbar_arrive(smem_addr(&sm.vfull[vslot]));
        sm.misc[18 + role] = drafts;
        sm.lkind[ls] = 1;  // released by the arrive below
        mbar_arrive(lbar);
      }
    } else {
      // The codes: K boxes from lanes 0..15, V boxes from lanes 16..31, rows at 128 bytes in order.
      if (lane == 0) {
        sm.lkind[ls] = 0;  // released by the arrive below
        mbar_arrive_expect_tx(lbar, 2 * tb.bytes);
      }
      __syncwarp();
      uint8_t* dst = sm.land + static_cast<size_t>(ls) * kLandBytes + kv * (kLandBytes / 2);
      if (i < tb.nbox) tma_load_2d(smem_addr(dst) + tb.off, kv ? &maps.tv : &maps.tk, 0, tb.y, lbar, policy);
    }
    ++issued;
    if (lane == 0) sm.misc[12 + role] = issued;
  }
}

// ============================================================ paired row blocks
//
// Stacks of 129..256 rows per KV head (whole-tree and whole-chain query modes):
// a unit holds two 128-row blocks of one KV head, so each K/V tile leaves HBM
// once for both.  Warpgroup w owns block w on every tile: S_w = Q_w K^T into
// its own two S buffers, its own online softmax, O_w += P_w V into its own
// accumulator and its own epilogue (no merge between the warpgroups).
// TMEM: S_{w,j} (tile parity j) at columns 64 (2 w + j), O_w at 256 + 128 w.
// P stays in tensor memory: the softmax writes P_w (bf16 pairs, 32 columns)
// over the S columns it has read, and P.V takes its A operand from there, so
// the softmax of the next tile never waits for this tile's P.V, and S buffer
// (w, j) is released when P.V of its tile completes.

struct SmemPair {
  uint8_t* kring;      // kPairNK x K tile
  uint8_t* vring;      // kPairNV x V tile
  uint8_t* qbuf;       // Q_0, Q_1 (kQBufBytes each)
  uint64_t* kfull;     // [kPairNK]  TMA -> QK^T issuer
  uint64_t* kempty;    // [kPairNK]  both QK^T of the tile completed -> TMA (one commit per issuing thread)
  uint64_t* vfull;     // [kPairNV]  TMA -> P.V issuer (and warpgroup 0 on partial tiles)
  uint64_t* vempty;    // [kPairNV]  both P.V of the tile completed -> TMA (one commit per issuing thread)
  uint64_t* qfull;     // [1]
  uint64_t* qempty;    // [1]
  uint64_t* sfull;     // [4]  S_{w,j} written (index 2 w + j)
  uint64_t* sfree;     // [4]  P.V of the tile in S_{w,j} completed: the buffer is free
  uint64_t* pfull;     // [4]  P_w of a tile with parity j written over S_{w,j} (128 threads)
  uint64_t* ofree;     // [2]  warpgroup w's epilogue read O_w (128 threads)
  uint64_t* mmadone;   // [4]  every MMA of an issuing thread completed (QK^T 0, 1, P.V 0, 1)
  uint64_t* anc;       // [64]
  int* par;            // [64]
  uint32_t* tmem_base;
  int* misc;           // as Smem::misc
  int* len;
  int* base;
};

__host__ __device__ inline size_t smem_bytes_pair(int C) {
  size_t off = static_cast<size_t>(kPairNK + kPairNV) * kKVBytes + 2 * kQBufBytes;
  off += sizeof(uint64_t) * (2 * kPairNK + 2 * kPairNV + 2 + 4 + 4 + 4 + 2 + 4);
  off += sizeof(uint64_t) * kMaxTreeNodes + sizeof(int) * kMaxTreeNodes;
  off += sizeof(uint32_t) * 4 + sizeof(int) * kMiscInts;
  off += sizeof(int) * (2 * C + 1);
  return off + 1024;
}

__device__ SmemPair carve_pair(uint8_t* raw, int C) {
  SmemPair s;
  uint8_t* p = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  s.kring = p;
  p += kPairNK * kKVBytes;
  s.vring = p;
  p += kPairNV * kKVBytes;
  s.qbuf = p;
  p += 2 * kQBufBytes;
  uint64_t* b = reinterpret_cast<uint64_t*>(p);
  s.kfull = b;
  s.kempty = s.kfull + kPairNK;
  s.vfull = s.kempty + kPairNK;
  s.vempty = s.vfull + kPairNV;
  s.qfull = s.vempty + kPairNV;
  s.qempty = s.qfull + 1;
  s.sfull = s.qempty + 1;
  s.sfree = s.sfull + 4;
  s.pfull = s.sfree + 4;
  s.ofree = s.pfull + 4;
  s.mmadone = s.ofree + 2;
  s.anc = s.mmadone + 4;
  s.par = reinterpret_cast<int*>(s.anc + kMaxTreeNodes);
  s.tmem_base = reinterpret_cast<uint32_t*>(s.par + kMaxTreeNodes);
  s.misc = reinterpret_cast<int*>(s.tmem_base + 4);
  s.len = s.misc + kMiscInts;
  s.base = s.len + C;
  return s;
}

// S_w = Q_w K^T of every tile, for one block w (one issuing thread per block:
// MMAs into one accumulator run one after another, each waiting for the last,
// while those of the other block's thread overlap them; a commit tracks only
// its own thread's MMAs, so S_w is released as soon as its own chain is done).
// Tile t needs its K tile, the piece's q blocks (first tile of a piece) and S
// buffer (w, t & 1), freed by the completion of P.V of block w of tile t - 2.
__device__ __forceinline__ void run_mma_qk_pair(const AttnParams& p, const SmemPair& sm, const Pipe& pipe,
                                                uint32_t tmem, Cursor cu, int w) {
  constexpr uint32_t idesc = idesc_bf16(128, 64, false);
  int piece = 0;
  const uint32_t qbase = smem_addr(sm.qbuf + w * kQBufBytes);
  for (int t = 0; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int j = t & 1;
    bool ok = !*pipe.abort;
    if (ok && ti.first) ok = mbar_wait(smem_addr(sm.qfull), piece & 1, p.err, p.wait_ns);
    if (ok) ok = mbar_wait(smem_addr(&sm.kfull[t % kPairNK]), (t / kPairNK) & 1, p.err, p.wait_ns);
    if (ok && t >= 2) ok = mbar_wait(smem_addr(&sm.sfree[2 * w + j]), ((t - 2) >> 1) & 1, p.err, p.wait_ns);
    if (!ok) {
      *pipe.abort = 1;
      break;
    }
    if (ti.first) ++piece;
    if (w == 0) {
      if (ti.first) sm.misc[4] = piece;
      sm.misc[2] = t + 1;
    }
    tc_fence_after();
    const uint32_t kbase = smem_addr(sm.kring + static_cast<size_t>(t % kPairNK) * kKVBytes);
    const bool grouped = ti.draft || p.prefix_grouped;
    const uint32_t half_off = grouped ? kGroupHalfBytes : kHalfBytes, group_off = grouped ? kGroupBytes : 1024;
#pragma unroll
    for (int ks = 0; ks < kHeadDim / 16; ++ks) {
      const uint64_t a = smem_desc_sw128(qbase + (ks >> 2) * (kQRows * 128) + (ks & 3) * 32, 16, 1024);
      const uint64_t b = smem_desc_sw128(kbase + (ks >> 2) * half_off + (ks & 3) * 32, 16, group_off);
      tc_mma(tmem + (2 * w + j) * kTileKeys, a, b, idesc, ks > 0 ? 1u : 0u);
    }
    tc_commit(smem_addr(&sm.sfull[2 * w + j]));
    tc_commit(smem_addr(&sm.kempty[t % kPairNK]));  // completes with both blocks' commits
    if (ti.last) tc_commit(smem_addr(sm.qempty));   // likewise
  }
  tc_commit(smem_addr(&sm.mmadone[w]));
}

// O_w += P_w V of every tile, for one block w (one issuing thread per block),
// with P_w read from tensor memory (the S columns of the tile).  The first P.V
// into O_w of a piece (which overwrites O_w) needs the previous piece's
// epilogue to have read O_w.  Each completion frees S buffer (w, t & 1) for
// QK^T of tile t + 2 and tells the softmax that O_w holds P.V of tile t.
__device__ __forceinline__ void run_mma_pv_pair(const AttnParams& p, const SmemPair& sm, const Pipe& pipe,
                                                uint32_t tmem, Cursor cu, int w) {
  constexpr uint32_t idesc = idesc_bf16(128, 128, true);
  int piece = 0, piece_t0 = 0;
  const uint32_t o = tmem + kTmemO + 128 * w;
  for (int t = 0; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int j = t & 1;
    if (ti.first) {
      ++piece;
      piece_t0 = t;
    }
    bool ok = !*pipe.abort;
    if (ok) ok = mbar_wait(smem_addr(&sm.vfull[t % kPairNV]), (t / kPairNV) & 1, p.err, p.wait_ns);
    if (ok && t == piece_t0 && piece > 1) ok = mbar_wait(smem_addr(&sm.ofree[w]), (piece - 2) & 1, p.err, p.wait_ns);
    if (ok) ok = mbar_wait(smem_addr(&sm.pfull[2 * w + j]), (t >> 1) & 1, p.err, p.wait_ns);
    if (!ok) {
      *pipe.abort = 1;
      break;
    }
    if (w == 0) sm.misc[6] = t + 1;
    tc_fence_after();
    const uint32_t vbase = smem_addr(sm.vring + static_cast<size_t>(t % kPairNV) * kKVBytes);
    const bool grouped = ti.draft || p.prefix_grouped;
    const uint32_t half_off = grouped ? kGroupHalfBytes : kHalfBytes, group_off = grouped ? kGroupBytes : 1024;
    const uint32_t pcol = tmem + (2 * w + j) * kTileKeys;  // P_w: 32 columns of bf16 pairs
#pragma unroll
    for (int k16 = 0; k16 < kTileKeys / 16; ++k16) {
      const uint64_t bd = smem_desc_sw128(vbase + k16 * 2 * group_off, half_off, group_off);
      tc_mma_tmem_a(o, pcol + 8 * k16, bd, idesc, (t == piece_t0 && k16 == 0) ? 0u : 1u);
    }
    tc_commit(smem_addr(&sm.sfree[2 * w + j]));
    tc_commit(smem_addr(&sm.vempty[t % kPairNV]));  // completes with both blocks' commits
  }
  tc_commit(smem_addr(&sm.mmadone[2 + w]));
}

// Softmax and epilogue of warpgroup wg = block wg of every unit: thread =
// TMEM lane = row r of the block, all 64 S columns of a tile.
__device__ __forceinline__ void run_softmax_pair(const AttnParams& p, const SmemPair& sm, const Pipe& pipe,
                                                 uint32_t tmem, Cursor cu) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3, wg = warp >> 2;
  const int wtid = threadIdx.x & 127;
  const int r = quarter * 32 + lane;
  const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
  const uint32_t my_s = trow + 2 * wg * kTileKeys;  // S_{wg, j} at my_s + 64 j
  const uint32_t my_o = trow + kTmemO + 128 * wg;
  const int HR = p.hkv * p.row_blocks;
  const float qscale = p.qscale;
  const bool tree = p.tree != 0;
  const int nq = p.Nq, n_nodes = p.N;
  int unit_c = -1, unit_hr = -1, h = 0, rr = 0, nl = 0;
  bool valid = false, warp_live = false;
  float m_run = -INFINITY, l_run = 0.f;
  int anc_seq = -1;
  wait_for_prerequisite_grid();
  for (int t = 0; cu.t < cu.t_end; ++t, cursor_next(cu, p, sm.len)) {
    const TileInfo ti = tile_info(cu, p);
    const int j = t & 1;
    if (cu.c != unit_c || cu.hr != unit_hr) {
      unit_c = cu.c;
      unit_hr = cu.hr;
      h = cu.hr / p.row_blocks;
      const int rb = cu.hr - h * p.row_blocks;
      const int row0 = rb * p.rows_per_unit + wg * kQRows;  // this warpgroup's first stacked row
      rr = row0 + r;
      valid = rr < p.rows_total;
      warp_live = row0 + quarter * 32 < p.rows_total;
      nl = valid ? rr / p.G : 0;
    }
    if (ti.first) {
      m_run = -INFINITY;
      l_run = 0.f;
    }
    if (ti.draft && tree) {
      const int seq = cu.c / (p.C / p.B);
      if (seq != anc_seq) {
        build_ancestor_masks(p, seq, sm.anc, sm.par, threadIdx.x, kSoftmaxThreads, kBarSoftmax);
        anc_seq = seq;
      }
    }
    bool live = !*pipe.abort;
    if (live && !mbar_wait(smem_addr(&sm.sfull[2 * wg + j]), (t >> 1) & 1, p.err, p.wait_ns)) {
      *pipe.abort = 1;
      live = false;
    }
    live = __all_sync(0xffffffffu, live);
    tc_fence_after();
    float pr[kTileKeys];
    bool any_rescale = false;
    float alpha = 1.f;
    if (live && warp_live) {
      uint32_t sv[kTileKeys];
      tmem_ld32(my_s + j * kTileKeys, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
      tmem_ld32(my_s + j * kTileKeys + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
      tmem_wait_ld();
      // pr holds the raw scores; the scale is folded into the exponent's argument (row_exp),
      // 2^(s qscale - m) = ex2(fma(s, qscale, -m)), and the row max is taken on the raw scores
      // (qscale > 0; row_max): fewer instructions per score (whole-tree hybrid tree 99.4 -> 94.5 us
      // per call for the folded scale alone).
      if (valid && !ti.draft && ti.nkeys >= kTileKeys) {  // a full prefix tile: every key is visible
#pragma unroll
        for (int k = 0; k < kTileKeys; ++k) pr[k] = __uint_as_float(sv[k]);
      } else {
        uint64_t vis = 0;
        if (valid) {
          vis = ti.nkeys >= 64 ? ~0ull : ((1ull << ti.nkeys) - 1ull);
          if (ti.draft) {
            uint64_t dm;
            if (tree) {
              dm = sm.anc[min(nl, nq - 1)] >> ti.key0;  // tree drafts have N <= 64, so key0 == 0
            } else {
              const int last = n_nodes - nq + nl - ti.key0;  // chain: slots key0 .. node are visible
              dm = last >= 63 ? ~0ull : (last < 0 ? 0ull : ((2ull << last) - 1ull));
            }
            vis &= dm;
          }
        }
#pragma unroll
        for (int k = 0; k < kTileKeys; ++k) pr[k] = ((vis >> k) & 1u) ? __uint_as_float(sv[k]) : -INFINITY;
      }
      const float mx = row_max(pr) * qscale;
      // Lazy rescale: move this row's reference max only when it grows by > 2^8.
      const bool grow = valid && (m_run == -INFINITY ? mx != -INFINITY : mx > m_run + kRescaleThreshold);
      const bool rescale_o = grow && m_run != -INFINITY;
      any_rescale = __any_sync(0xffffffffu, rescale_o);
      alpha = rescale_o ? ex2(m_run - mx) : 1.f;
      l_run *= alpha;
      if (grow) m_run = mx;
      const float m_use = m_run == -INFINITY ? 0.f : m_run;
      uint32_t pk[kTileKeys / 2];  // P as bf16 pairs (rows past the stack hold zeros)
      l_run += row_exp<kTileKeys, false>(pr, qscale, m_use, 1.f, pk);
      tmem_st32(my_s + j * kTileKeys, pk);  // P over the S columns just read
    }
    // Only a rescale of O_wg waits for P.V of the previous tile (sfree of its S buffer, which P.V
    // commits when it completes); P of this tile is released without it, so that hand-off stays off
    // the loop through the S buffers (whole-tree hybrid tree 83.3 -> 77.4 us per call on GB300).  A
    // rescale needs an earlier tile of the piece, so t >= 1, and the wait is unambiguous: P.V of
    // tile t - 3 completed before QK^T of tile t - 1 was issued, and P.V of tile t + 1 cannot
    // complete before the pfull of tile t + 1.
    if (live && warp_live) {
      if (any_rescale) {  // O_wg *= alpha (P.V of this tile is issued only after pfull below)
        if (!mbar_wait(smem_addr(&sm.sfree[2 * wg + ((t - 1) & 1)]), ((t - 1) >> 1) & 1, p.err, p.wait_ns))
          *pipe.abort = 1;
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          tmem_ld32(my_o + 32 * c, o);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 32; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * alpha);
          tmem_st32(my_o + 32 * c, o);
        }
      }
      tmem_wait_st();
    }
    if (live && ti.nkeys < kTileKeys) {
      // V rows past the valid keys may hold NaN; 0 * NaN would poison P.V.  Each warpgroup clears them
      // before it releases its P (P.V of block w is issued after P_w alone; both write the same zeros).
      if (!mbar_wait(smem_addr(&sm.vfull[t % kPairNV]), (t / kPairNV) & 1, p.err, p.wait_ns)) *pipe.abort = 1;
      uint8_t* vptr = sm.vring + static_cast<size_t>(t % kPairNV) * kKVBytes;
      const bool grouped = ti.draft || p.prefix_grouped;
      const int nz = (kTileKeys - ti.nkeys) * 16;
      for (int i = wtid; i < nz; i += kQRows) {
        const int key = ti.nkeys + (i >> 4), ch = i & 15;
        *reinterpret_cast<uint4*>(vptr + tile_off_tc(key, ch, grouped)) = make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
    }
    tc_fence_before();
    mbar_arrive(smem_addr(&sm.pfull[2 * wg + j]));
    if (ti.last) {
      // Every P.V of the piece has completed once P.V of tile t has (they complete in order; the
      // parity is unambiguous as for the rescale wait above).
      bool ok = live && mbar_wait(smem_addr(&sm.sfree[2 * wg + (t & 1)]), (t >> 1) & 1, p.err, p.wait_ns);
      ok = __all_sync(0xffffffffu, ok);
      tc_fence_after();
      if (ok && warp_live) {
        const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
        const float lse2 = l_run > 0.f ? m_run + __log2f(l_run) : -INFINITY;
        const bool whole = cu.lt == cu.ut - 1 && (cu.t - cu.t_begin) >= cu.lt;
        const int slot = cu.c * HR + cu.hr + blockIdx.x;
        const int urow = wg * kQRows + r;  // row within the unit
        size_t orow = 0;
        if (valid && whole) {
          const int g = rr - nl * p.G;
          orow = (static_cast<size_t>(cu.c) * p.Nq + nl) * p.hq + h * p.G + g;
        }
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          tmem_ld32(my_o + 32 * c, o);
          tmem_wait_ld();
          if (valid) {
            if (whole) {
              uint4* dst = reinterpret_cast<uint4*>(p.out + orow * kHeadDim + 32 * c);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                uint4 w4;
                w4.x = pack_bf16x2(__uint_as_float(o[8 * k + 0]) * inv, __uint_as_float(o[8 * k + 1]) * inv);
                w4.y = pack_bf16x2(__uint_as_float(o[8 * k + 2]) * inv, __uint_as_float(o[8 * k + 3]) * inv);
                w4.z = pack_bf16x2(__uint_as_float(o[8 * k + 4]) * inv, __uint_as_float(o[8 * k + 5]) * inv);
                w4.w = pack_bf16x2(__uint_as_float(o[8 * k + 6]) * inv, __uint_as_float(o[8 * k + 7]) * inv);
                dst[k] = w4;
              }
            } else {
              float4* dst = reinterpret_cast<float4*>(
                  p.ws_o + (static_cast<size_t>(slot) * p.rows_per_unit + urow) * kHeadDim + 32 * c);
#pragma unroll
              for (int k = 0; k < 8; ++k)
                dst[k] = make_float4(__uint_as_float(o[4 * k]) * inv, __uint_as_float(o[4 * k + 1]) * inv,
                                     __uint_as_float(o[4 * k + 2]) * inv, __uint_as_float(o[4 * k + 3]) * inv);
            }
          }
        }
        if (valid) {
          if (whole) p.lse[orow] = lse2 * 0.69314718055994531f;
          else p.ws_lse[static_cast<size_t>(slot) * p.rows_per_unit + urow] = lse2;
        }
      }
      tc_fence_before();
      mbar_arrive(smem_addr(&sm.ofree[wg]));
    }
  }
}

__global__ void __launch_bounds__(kPairThreads, 1)
    attn_tc_pair_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ TensorMaps maps, int nq_box) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();  // the merge may be scheduled as CTAs finish
  const int len0 = static_cast<int>(threadIdx.x) < p.C ? p.seq_lens[threadIdx.x] : -1;
  const SmemPair sm = carve_pair(smem_raw, p.C);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kPairNK; ++s) {
      mbar_init(smem_addr(&sm.kfull[s]), 1);
      mbar_init(smem_addr(&sm.kempty[s]), 2);  // one commit per QK^T issuer
    }
    for (int s = 0; s < kPairNV; ++s) {
      mbar_init(smem_addr(&sm.vfull[s]), 1);
      mbar_init(smem_addr(&sm.vempty[s]), 2);  // one commit per P.V issuer
    }
    mbar_init(smem_addr(sm.qfull), 1);
    mbar_init(smem_addr(sm.qempty), 2);
    for (int b = 0; b < 4; ++b) {
      mbar_init(smem_addr(&sm.sfull[b]), 1);
      mbar_init(smem_addr(&sm.sfree[b]), 1);
      mbar_init(smem_addr(&sm.pfull[b]), kQRows);
      mbar_init(smem_addr(&sm.mmadone[b]), 1);
    }
    for (int w = 0; w < 2; ++w) mbar_init(smem_addr(&sm.ofree[w]), kQRows);
    for (int i = 0; i < kMiscInts; ++i) sm.misc[i] = 0;
    fence_mbar_init();
    prefetch_tensormap(&maps.tk);
    prefetch_tensormap(&maps.tv);
    prefetch_tensormap(&maps.dk);
    prefetch_tensormap(&maps.dv);
    prefetch_tensormap(&maps.q);
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_addr(sm.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  build_plan(p, sm.len, sm.base, len0);  // block-wide barriers inside
  tc_fence_after();
  const uint32_t tmem = *sm.tmem_base;
  const Cursor cu = cursor_begin(p, sm.len, sm.base);
  Pipe pipe{nullptr, nullptr, nullptr, 0, reinterpret_cast<volatile int*>(&sm.misc[0]), nullptr};
  if (warp == kProducerWarp || warp == kProducerVWarp) {
    run_producer_tc<kModePair>(p, maps, sm, pipe, cu, nq_box, warp == kProducerWarp ? 0 : 1);
  } else if (warp == kMmaWarp || warp == kMmaPvWarp || warp == kMmaWarp1 || warp == kMmaPvWarp1) {
    // One QK^T and one P.V issuer per block: warps 11, 8 for block 0 and 12, 13 for block 1.
    const int w = (warp == kMmaWarp1 || warp == kMmaPvWarp1) ? 1 : 0;
    const bool qk = warp == kMmaWarp || warp == kMmaWarp1;
    if ((threadIdx.x & 31) == 0 && cu.t < cu.t_end) {
      if (qk) run_mma_qk_pair(p, sm, pipe, tmem, cu, w);
      else run_mma_pv_pair(p, sm, pipe, tmem, cu, w);
      // Every MMA must have completed before TMEM is released (retried, bounded, as in attn_tc_kernel).
      const int done = qk ? w : 2 + w;
      for (int k = 0; k < 4 && !mbar_wait(smem_addr(&sm.mmadone[done]), 0, p.err); ++k) {
      }
    }
    __syncwarp();
  } else if (warp < 8) {
    run_softmax_pair(p, sm, pipe, tmem, cu);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0 && *pipe.abort) {
    // A wait timed out: let every TMA load still in flight land before the CTA exits.
    for (int k = sm.misc[2]; k < max(sm.misc[8], sm.misc[9]); ++k)
      if (k < sm.misc[8 + (k & 1)] && !mbar_wait(smem_addr(&sm.kfull[k % kPairNK]), (k / kPairNK) & 1, p.err)) break;
    for (int k = sm.misc[6]; k < max(sm.misc[10], sm.misc[11]); ++k)
      if (k < sm.misc[10 + (k & 1)] && !mbar_wait(smem_addr(&sm.vfull[k % kPairNV]), (k / kPairNV) & 1, p.err)) break;
    for (int k = sm.misc[4]; k < sm.misc[3]; ++k)
      if (!mbar_wait(smem_addr(sm.qfull), k & 1, p.err)) break;
  }
  if (warp == kMmaWarp) tmem_dealloc(tmem, kTmemCols);
}

template <bool kSpread, bool kF8>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ AttnParams p, const __grid_constant__ TensorMaps maps, int nq_box) {
  constexpr int NK = kF8 ? kF8NK : kNK, NV = kF8 ? kF8NV : kNV;
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) allow_dependent_launch();  // the merge may be scheduled as CTAs finish
  // The plan's lengths are loaded first, so that their latency overlaps the set-up below
  // (a negative length, invalid anyway, is clamped by the ordinary path).
  const int len0 = static_cast<int>(threadIdx.x) < p.C ? p.seq_lens[threadIdx.x] : -1;
  const Smem sm = carve(smem_raw, p.C, kF8);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 32 && p.paged) {
    // The page-table line of this CTA's first tile, were every length at its bound (exact
    // for equal lengths; a mere extra prefetch otherwise), is brought into L2 meanwhile.
    const int HR = p.hkv * p.row_blocks;
    const long long ut = (p.len_bound + kTileKeys - 1) / kTileKeys + p.draft_tiles;
    const long long T = static_cast<long long>(p.C) * HR * ut;
    const long long t0 = static_cast<long long>(blockIdx.x) * ((T + p.num_ctas - 1) / p.num_ctas);
    const long long c = t0 / (HR * ut), lt = (t0 - c * HR * ut) % ut;
    const long long pg = lt * kTileKeys / p.page_size;
    if (c < p.C && lt * kTileKeys < p.len_bound && pg < p.max_pages)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(p.page_table + c * p.max_pages + pg));
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < NK; ++s) {
      mbar_init(smem_addr(&sm.kfull[s]), 1);
      mbar_init(smem_addr(&sm.kempty[s]), 1);
    }
    for (int s = 0; s < NV; ++s) {
      mbar_init(smem_addr(&sm.vfull[s]), 1);
      mbar_init(smem_addr(&sm.vempty[s]), 1);
    }
    mbar_init(smem_addr(sm.qfull), 1);
    mbar_init(smem_addr(sm.qempty), 1);
    for (int b = 0; b < kNS; ++b) {
      mbar_init(smem_addr(&sm.sfull[b]), 1);
      mbar_init(smem_addr(&sm.sfree[b]), 1);
      mbar_init(smem_addr(&sm.pfull[b]), kSoftmaxThreads / 2);
    }
    if constexpr (kF8) {
      for (int l = 0; l < kLandSlots; ++l) {
        mbar_init(smem_addr(&sm.lfull[l]), 1);
        mbar_init(smem_addr(&sm.lfree[l]), 1);
      }
      mbar_init(smem_addr(sm.qland), 1);
      mbar_init(smem_addr(&sm.dland[0]), 1);
      mbar_init(smem_addr(&sm.dland[1]), 1);
    }
    mbar_init(smem_addr(sm.ofree), kSoftmaxThreads);
    mbar_init(smem_addr(&sm.mmadone[0]), 1);
    mbar_init(smem_addr(&sm.mmadone[1]), 1);
    for (int i = 0; i < kMiscInts; ++i) sm.misc[i] = 0;
    fence_mbar_init();
    prefetch_tensormap(&maps.tk);
    prefetch_tensormap(&maps.tv);
    prefetch_tensormap(&maps.dk);
    prefetch_tensormap(&maps.dv);
    prefetch_tensormap(&maps.q);
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_addr(sm.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  build_plan(p, sm.len, sm.base, len0);  // block-wide barriers inside
  tc_fence_after();
  const uint32_t tmem = *sm.tmem_base;
  const Cursor cu = cursor_begin(p, sm.len, sm.base);
  Pipe pipe{nullptr, nullptr, nullptr, 0, reinterpret_cast<volatile int*>(&sm.misc[0]), nullptr};
  if (warp == kProducerWarp || warp == kProducerVWarp) {
    if constexpr (kF8) run_producer_f8(p, maps, sm, pipe, cu, nq_box, warp == kProducerWarp ? 0 : 1);
    else run_producer_tc<kSpread ? kModeSpread : kModeDense>(p, maps, sm, pipe, cu, nq_box, warp == kProducerWarp ? 0 : 1);
  } else if (warp == kMmaWarp || warp == kMmaPvWarp) {
    const int stream = warp == kMmaWarp ? 0 : 1;
    if ((threadIdx.x & 31) == 0 && cu.t < cu.t_end) {
      if (stream == 0) run_mma_qk<kF8>(p, sm, pipe, tmem, cu);
      else run_mma_pv<kF8>(p, sm, pipe, tmem, cu);
      // Every MMA must have completed before TMEM is released.  Each MMA issued reads shared memory
      // whose loads it already waited for, so it finishes; the wait is retried (bounded) if it runs
      // past its limit rather than freeing TMEM under a running MMA.
      for (int k = 0; k < 4 && !mbar_wait(smem_addr(&sm.mmadone[stream]), 0, p.err); ++k) {
      }
    }
    __syncwarp();
  } else if (warp < 8) {
    run_softmax<kSpread, kF8>(p, sm, pipe, tmem, cu);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0 && *pipe.abort) {
    // A wait timed out: let every TMA load still in flight land before the CTA exits.
    // Tile k was loaded by producer warp k % 2, which issues its tiles in order.
    for (int k = sm.misc[2]; k < max(sm.misc[8], sm.misc[9]); ++k)
      if (k < sm.misc[8 + (k & 1)] && !mbar_wait(smem_addr(&sm.kfull[k % NK]), (k / NK) & 1, p.err)) break;
    for (int k = sm.misc[6]; k < max(sm.misc[10], sm.misc[11]); ++k)
      if (k < sm.misc[10 + (k & 1)] && !mbar_wait(smem_addr(&sm.vfull[k % NV]), (k / NV) & 1, p.err)) break;
    if constexpr (!kF8) {
      for (int k = sm.misc[4]; k < sm.misc[3]; ++k)
        if (!mbar_wait(smem_addr(sm.qfull), k & 1, p.err)) break;
    } else {
      // q blocks, fp8 codes and draft tiles landed by the producer warps but not converted.
      for (int k = sm.misc[1]; k < sm.misc[3]; ++k)
        if (!mbar_wait(smem_addr(sm.qland), k & 1, p.err)) break;
      for (int role = 0; role < 2; ++role) {
        for (int j = sm.misc[14 + role]; j < sm.misc[12 + role]; ++j) {  // tile role + 2 j
          const int y = role + 2 * j;
          if (!mbar_wait(smem_addr(&sm.lfull[y % kLandSlots]), (y / kLandSlots) & 1, p.err)) break;
        }
        for (int j = sm.misc[18 + role]; j < sm.misc[16 + role]; ++j)
          if (!mbar_wait(smem_addr(&sm.dland[role]), j & 1, p.err)) break;
      }
    }
  }
  if (warp == kMmaWarp) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

cudaError_t attn_tc_occupancy(int C, int* ctas_per_sm) {
  const size_t smem = smem_bytes(C, false);
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, attn_tc_kernel<false, false>, kThreads, smem);
}

cudaError_t launch_attn_tc(const AttnParams& p, const TensorMaps& maps, int nq_box, bool spread, bool pair, bool pdl,
                           cudaStream_t stream) {
  if (pair) {
    const size_t smem = smem_bytes_pair(p.C);
    cudaError_t e = cudaFuncSetAttribute(attn_tc_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    return launch_maybe_pdl(attn_tc_pair_kernel, dim3(p.num_ctas), dim3(kPairThreads), smem, pdl, stream, p, maps,
                            nq_box);
  }
  const bool f8 = p.fp8 != 0;
  const size_t smem = smem_bytes(p.C, f8);
  auto* kernel = f8 ? (spread ? attn_tc_kernel<true, true> : attn_tc_kernel<false, true>)
                    : (spread ? attn_tc_kernel<true, false> : attn_tc_kernel<false, false>);
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch_maybe_pdl(kernel, dim3(p.num_ctas), dim3(kThreads), smem, pdl, stream, p, maps, nq_box);
}

}  // namespace kvshot
