// kvshot_attn_common.cuh -- device building blocks shared by the draft
// attention kernels: PTX wrappers, the bounded mbarrier wait, the stream-K
// tile cursor, the draft-tree ancestor masks and the TMA producer warp.
#pragma once

#include "kvshot_internal.h"

namespace kvshot {
namespace dev {
namespace {  // internal linkage: every translation unit gets its own copy

// ---------------------------------------------------------------- PTX wrappers

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void set_error(int32_t* err, int code) {
  if (err != nullptr) atomicCAS(err, 0, code);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Orders this thread's generic-proxy shared-memory accesses before later
// async-proxy (TMA) accesses to the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}

// Every wait gives up after a time limit, records KVSHOT_ERR_TIMEOUT and lets
// the kernel wind down instead of spinning forever.  The attention kernels'
// pipeline waits take the call's limit (AttnParams::wait_ns); waits for work
// already issued (the drain of in-flight copies after an abort, the last
// tensor-core operations before TMEM is freed) and the other kernels' waits
// take kWaitLimitNs.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Limits below this are polled with the non-blocking test and a timer check
// on every iteration (mbarrier.try_wait may suspend the thread for longer than
// such a limit, so the timer would never be looked at in time).
constexpr uint64_t kPollBelowNs = 100000;

// Non-blocking test of a phase's completion.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}

// Out-of-line part of every wait.  Below kPollBelowNs (a test limit) it polls the non-blocking test
// and the clock; otherwise it blocks in mbarrier.try_wait and looks at the clock every 64 tries.
__device__ __noinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity, int32_t* err, uint64_t limit_ns) {
  const uint64_t t0 = global_timer_ns();
  if (limit_ns < kPollBelowNs) {
    for (;;) {
      if (mbar_test_wait(bar, parity)) return true;
      if (global_timer_ns() - t0 > limit_ns) break;
    }
  } else {
    for (;;) {
      for (int i = 0; i < 64; ++i)
        if (mbar_try_wait(bar, parity)) return true;
      if (global_timer_ns() - t0 > limit_ns) break;
    }
  }
  set_error(err, KVSHOT_ERR_TIMEOUT);
  return false;
}

// The inline part is one non-blocking test: a phase already complete costs no call, and every wait
// that has to wait goes to the out-of-line slow path, which holds the limit logic.  (A blocking first
// probe could sit out a short limit; an inline limit check made every wait site larger and cost the
// attention kernels 10-15% on GB300.)
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int32_t* err,
                                          uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_test_wait(bar, parity)) return true;
  return mbar_wait_slow(bar, parity, err, limit_ns);
}

// Programmatic dependent launch.  The attention kernels let the kernel that
// follows them in the stream (the split merge, launched with programmatic
// stream serialization) be scheduled onto SMs as attention CTAs finish; that
// kernel waits for the whole attention grid to complete, memory included,
// before it reads anything, so only the launch latency is hidden.
__device__ __forceinline__ void allow_dependent_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void wait_for_prerequisite_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// 2-D tiled TMA load (box {64 elements, rows}) into 128B-swizzled shared memory.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}

// 3-D tiled TMA load with an L2 cache hint.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar), "l"(policy)
      : "memory");
}

// 4-D tiled TMA load with an L2 cache hint.
__device__ __forceinline__ void tma_load_4d_hint(uint32_t dst, const CUtensorMap* map, int x, int y, int z, int w,
                                                 uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(bar), "l"(policy)
      : "memory");
}

// 4-D tiled TMA load (default L2 policy).
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, int w,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void named_barrier_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                            uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                                  uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D += A * B, m16n8k16, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset, inside one K or V tile, of 16-byte chunk `ch` (0..15, i.e.
// dims 8ch..8ch+7) of key row r.  The tile is two 64-dim halves of TK rows of
// 128 bytes; TMA's 128-byte swizzle XORs the chunk index (mod 8) with the row
// index (mod 8).  Every 8-row group starts on a 1024-byte boundary.
__device__ __forceinline__ uint32_t tile_off(int r, int ch) {
  return static_cast<uint32_t>((ch >> 3) * kHalfBytes + r * 128 + (((ch & 7) ^ (r & 7)) << 4));
}

// The same offset for a tile in either layout, given the strides of its 8-row
// groups and of its 64-dim halves: {1024, kHalfBytes} for the halves layout
// above, {kGroupBytes, kGroupHalfBytes} for the grouped layout (8-row groups of
// both halves, as a grouped box lands).  The swizzle is the same in both.
struct TileLayout {
  uint32_t group, half;
};
__host__ __device__ constexpr TileLayout tile_layout(bool grouped) {
  return grouped ? TileLayout{kGroupBytes, kGroupHalfBytes} : TileLayout{1024u, static_cast<uint32_t>(kHalfBytes)};
}
__device__ __forceinline__ uint32_t tile_off(int r, int ch, TileLayout l) {
  if (l.group == 1024u && l.half == static_cast<uint32_t>(kHalfBytes)) return tile_off(r, ch);
  return static_cast<uint32_t>(r >> 3) * l.group + static_cast<uint32_t>(ch >> 3) * l.half +
         static_cast<uint32_t>(((r & 7) << 7) + (((ch & 7) ^ (r & 7)) << 4));
}

// ------------------------------------------------------------ work plan

// Clamped prefix length of cache c; out-of-range values are reported.
__device__ __forceinline__ int clamp_len(const AttnParams& p, int c) {
  int L = p.seq_lens[c];
  if (L < 0 || L > p.len_bound) {
    set_error(p.err, KVSHOT_ERR_DEVICE_BOUNDS);
    L = L < 0 ? 0 : p.len_bound;
  }
  return L;
}

// Clamped prefix length of cache c from its already loaded entry.
__device__ __forceinline__ int clamp_len_of(const AttnParams& p, int L) {
  if (L < 0 || L > p.len_bound) {
    set_error(p.err, KVSHOT_ERR_DEVICE_BOUNDS);
    L = L < 0 ? 0 : p.len_bound;
  }
  return L;
}

// s_len[c] = clamped L_c; s_base[c] = first global tile of cache c (prefix sum of
// units x tiles per unit).  Whole block participates.  `len0` may hold
// seq_lens[threadIdx.x], loaded early by the caller (-1: not loaded).
__device__ __forceinline__ void build_plan(const AttnParams& p, int* s_len, int* s_base, int len0 = -1) {
  const int HR = p.hkv * p.row_blocks;
  for (int c = threadIdx.x; c < p.C; c += blockDim.x) {
    const int L = (c == static_cast<int>(threadIdx.x) && len0 >= 0) ? clamp_len_of(p, len0) : clamp_len(p, c);
    s_len[c] = L;
    s_base[c + 1] = ((L + kTileKeys - 1) / kTileKeys + p.draft_tiles) * HR;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int carry = 0;
    for (int c0 = 0; c0 < p.C; c0 += 32) {
      const int c = c0 + lane;
      int v = c < p.C ? s_base[c + 1] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += t;
      }
      if (c < p.C) s_base[c + 1] = v + carry;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
    if (lane == 0) s_base[0] = 0;
  }
  __syncthreads();
}

// Tiles of CTA b: [b * tpc, min(T, (b + 1) * tpc)).
__device__ __forceinline__ int tiles_per_cta(int total, int ctas) { return (total + ctas - 1) / ctas; }

struct Cursor {
  int t, t_begin, t_end;  // global tile index and this CTA's range
  int c, hr, lt;          // cache, KV head x row block, tile within the unit
  int L, pt, ut;          // prefix length, prefix tiles, tiles per unit
};

__device__ __forceinline__ void cursor_load_cache(Cursor& cu, const AttnParams& p, const int* s_len) {
  cu.L = s_len[cu.c];
  cu.pt = (cu.L + kTileKeys - 1) / kTileKeys;
  cu.ut = cu.pt + p.draft_tiles;
}

__device__ __forceinline__ Cursor cursor_begin(const AttnParams& p, const int* s_len, const int* s_base) {
  Cursor cu;
  const int total = s_base[p.C];
  const int tpc = tiles_per_cta(total, p.num_ctas);
  cu.t_begin = cu.t = min(total, blockIdx.x * tpc);
  cu.t_end = min(total, cu.t + tpc);
  cu.c = 0;
  cu.hr = 0;
  cu.lt = 0;
  cu.L = cu.pt = cu.ut = 0;
  if (cu.t >= cu.t_end) return cu;
  int lo = 0, hi = p.C - 1;  // last cache whose first tile is <= t
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_base[mid] <= cu.t) lo = mid;
    else hi = mid - 1;
  }
  cu.c = lo;
  cursor_load_cache(cu, p, s_len);
  const int rem = cu.t - s_base[lo];
  cu.hr = rem / cu.ut;
  cu.lt = rem - cu.hr * cu.ut;
  return cu;
}

__device__ __forceinline__ void cursor_next(Cursor& cu, const AttnParams& p, const int* s_len) {
  ++cu.t;
  if (++cu.lt == cu.ut) {
    cu.lt = 0;
    if (++cu.hr == p.hkv * p.row_blocks) {
      cu.hr = 0;
      ++cu.c;
      if (cu.t < cu.t_end) cursor_load_cache(cu, p, s_len);
    }
  }
}

struct TileInfo {
  bool draft;   // draft tile (else prefix tile)
  int key0;     // first key: prefix token index, or draft slot
  int nkeys;    // valid keys in the tile (1..TK)
  bool first;   // first tile of this CTA's piece of the unit
  bool last;    // last tile of this CTA's piece of the unit
};

__device__ __forceinline__ TileInfo tile_info(const Cursor& cu, const AttnParams& p) {
  TileInfo ti;
  ti.draft = cu.lt >= cu.pt;
  ti.key0 = (ti.draft ? cu.lt - cu.pt : cu.lt) * kTileKeys;
  ti.nkeys = min(kTileKeys, (ti.draft ? p.N : cu.L) - ti.key0);
  ti.first = (cu.t == cu.t_begin) || cu.lt == 0;
  ti.last = (cu.t == cu.t_end - 1) || cu.lt == cu.ut - 1;
  return ti;
}

// ------------------------------------------------------ draft-tree masks

// s_anc[nl] = bitmask of draft slots visible to query node N - Nq + nl: the
// node itself and its ancestors (tree verification mask).  Built by the
// `nthreads` consumer threads (tid in [0, nthreads)), which must all call it;
// two named barriers (id `bar`) fence it.  Invalid parents are reported and
// treated as roots.
__device__ __forceinline__ void build_ancestor_masks(const AttnParams& p, int seq, uint64_t* s_anc, int* s_par, int tid,
                                     int nthreads, int bar) {
  const int* par = p.tree_parent + static_cast<size_t>(seq) * p.N;
  for (int i = tid; i < p.N; i += nthreads) {
    int v = par[i];
    if (v < -1 || v >= i) {
      set_error(p.err, KVSHOT_ERR_TREE);
      v = -1;
    }
    s_par[i] = v;
  }
  named_barrier_sync(bar, nthreads);
  for (int nl = tid; nl < p.Nq; nl += nthreads) {
    uint64_t bits = 0;
    for (int m = p.N - p.Nq + nl; m >= 0; m = s_par[m]) bits |= 1ull << m;  // parents strictly decrease
    s_anc[nl] = bits;
  }
  named_barrier_sync(bar, nthreads);
}

// Is draft slot m visible to query row r (row of the unit's GQA stack)?
__device__ __forceinline__ bool draft_visible(const AttnParams& p, const uint64_t* s_anc, int r, int m) {
  if (m >= p.N) return false;
  const int nl = min(r / p.G, p.Nq - 1);
  if (p.tree) return (s_anc[nl] >> m) & 1ull;
  return m <= p.N - p.Nq + nl;
}

// ------------------------------------------------------------ TMA producer

// A page id checked against the pool; out-of-range ids are reported and replaced by page 0.
__device__ __forceinline__ int valid_page_id(const AttnParams& p, int pid) {
  if (pid < 0 || pid >= p.num_pages) {
    set_error(p.err, KVSHOT_ERR_DEVICE_BOUNDS);
    pid = 0;
  }
  return pid;
}

// Page ids of the producer warp, 32 consecutive page-table entries of one
// cache per load (lane i holds entry base + i, validated when loaded),
// double-buffered: while the current window is used the next one is already
// in flight.  The cache's first window is kept as well, since the KV heads of
// one cache (consecutive units) walk the same pages.
struct PageWindow {
  int cur_c = -1, cur_base = 0, cur_pid = 0;
  int nxt_c = -1, nxt_base = 0, nxt_pid = 0;
  int head_c = -1, head_pid = 0;

  __device__ __forceinline__ static int load(const AttnParams& p, int c, int base, int lane) {
    const int pg = base + lane;
    return pg < p.max_pages ? p.page_table[static_cast<size_t>(c) * p.max_pages + pg] : 0;
  }
  // Make pages [pg, pg + n) of cache c (n <= 32, windows stay aligned to the
  // tile's page count; the cache has `pages` pages in use) available in
  // cur_pid.  Only entries of pages in use are validated.  Warp-wide.
  __device__ __forceinline__ void cover(const AttnParams& p, int c, int pages, int pg, int n, int lane) {
    if (cur_c == c && pg >= cur_base && pg + n <= cur_base + 32) return;
    if (nxt_c == c && pg >= nxt_base && pg + n <= nxt_base + 32) {
      cur_c = nxt_c;
      cur_base = nxt_base;
      cur_pid = nxt_base + lane < pages ? valid_page_id(p, nxt_pid) : 0;
    } else if (pg == 0 && head_c == c) {
      cur_c = c;
      cur_base = 0;
      cur_pid = head_pid;
    } else {
      cur_c = c;
      cur_base = pg;
      cur_pid = load(p, c, pg, lane);
      cur_pid = pg + lane < pages ? valid_page_id(p, cur_pid) : 0;
      if (pg == 0) {
        head_c = c;
        head_pid = cur_pid;
      }
    }
    nxt_c = c;
    nxt_base = cur_base + 32;
    nxt_pid = load(p, c, nxt_base, lane);  // validated when it becomes current
  }
  // Page id of page pg (covered), broadcast to the warp.
  __device__ __forceinline__ int get(int pg) const { return __shfl_sync(0xffffffffu, cur_pid, pg - cur_base); }
};

struct Pipe {
  uint8_t* ring;       // stages x kStageBytes, 1024-aligned
  uint64_t* full;      // [stages] TMA -> consumers
  uint64_t* empty;     // [stages] consumers -> TMA
  int stages;
  volatile int* abort; // set when a wait timed out
  int* issued;         // tiles issued by the producer
};

// q staging (tensor-memory kernel only): piece k's query block goes to buffer
// k % nbuf (two 64-dim halves of 128 rows, 128B-swizzled).
struct QPipe {
  uint8_t* buf;        // nbuf x kQBufBytes, 1024-aligned
  uint64_t* full;      // [nbuf] TMA -> MMA issuer
  uint64_t* empty;     // [nbuf] MMA completion -> TMA
  int nbuf;            // q buffers (piece k uses buffer k % nbuf)
  int rows;            // rows loaded per box (G x nodes per box)
  int nq_box;          // draft nodes per box
  int* issued;         // q blocks issued
};
constexpr int kQRows = 128;
constexpr int kQBufBytes = 2 * kQRows * 128;

// The producer warp: walks this CTA's tiles and issues their TMA loads into the
// stage ring, one tile ahead on the page-table reads.  Lane 0 issues.
__device__ __forceinline__ void run_producer(const AttnParams& p, const TensorMaps& maps, const Pipe& pipe, const int* s_len,
                             Cursor cu, const QPipe* qp = nullptr) {
  const int lane = threadIdx.x & 31;
  const uint64_t policy = l2_policy_evict_first();
  int stage = 0;
  uint32_t phase = 0;
  int issued = 0;
  int piece = 0;
  PageWindow win;
  while (cu.t < cu.t_end) {
    const int h = cu.hr / p.row_blocks;
    const int L = cu.L;
    const bool draft = cu.lt >= cu.pt;
    const int key0 = (draft ? cu.lt - cu.pt : cu.lt) * kTileKeys;
    const int nkeys = min(kTileKeys, (draft ? p.N : L) - key0);
    // Page ids of this tile's boxes (box i covers rows key0 + i * box_rows).
    int pids[kTileKeys / 8];
    if (p.paged && !draft) {
      const int pg0 = key0 / p.page_size;
      const int npg = (nkeys + p.box_rows - 1) / p.box_rows;  // one box per page (or one box inside a page)
      win.cover(p, cu.c, (cu.L + p.page_size - 1) / p.page_size, pg0, p.box_rows < p.page_size ? 1 : npg, lane);
#pragma unroll
      for (int i = 0; i < kTileKeys / 8; ++i)
        pids[i] = win.get(pg0 + (p.box_rows < p.page_size ? 0 : min(i, npg - 1)));
    }

    int ok = 1;
    if (qp != nullptr && (cu.t == cu.t_begin || cu.lt == 0)) {
      // First tile of a piece: stage the unit's query block (all its G x Nq rows).
      if (lane == 0) {
        const int qb = piece % qp->nbuf;
        const uint32_t qbar = smem_addr(&qp->full[qb]);
        ok = mbar_wait(smem_addr(&qp->empty[qb]), ((piece / qp->nbuf) & 1) ^ 1u, p.err, p.wait_ns) ? 1 : 0;
        if (ok && !*pipe.abort) {
          const int rb = cu.hr - h * p.row_blocks;
          const uint32_t dst = smem_addr(qp->buf + qb * kQBufBytes);
          mbar_arrive_expect_tx(qbar, 2 * qp->rows * 128);
          tma_load_4d(dst, &maps.q, 0, h * p.G, rb * qp->nq_box, cu.c, qbar);
          tma_load_4d(dst + kQRows * 128, &maps.q, 64, h * p.G, rb * qp->nq_box, cu.c, qbar);
          *qp->issued = piece + 1;
        } else {
          ok = 0;
        }
      }
      ++piece;
    }
    if (lane == 0 && ok) {
      ok = mbar_wait(smem_addr(&pipe.empty[stage]), phase ^ 1u, p.err, p.wait_ns) ? 1 : 0;
      if (!ok || *pipe.abort) ok = 0;
    }
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) {
      if (lane == 0) *pipe.abort = 1;
      break;
    }
    {
      // Lane 0 posts the tile's byte count; every lane then issues at most one
      // box: box = lane -> (tensor K/V, 64-dim half, page or 8-row group).
      const uint32_t full_bar = smem_addr(&pipe.full[stage]);
      const uint32_t kdst = smem_addr(pipe.ring + static_cast<size_t>(stage) * kStageBytes);
      const int kv = lane & 1, hf = (lane >> 1) & 1, i = lane >> 2;
      const uint32_t dst = kdst + kv * kKVTileBytes + hf * kHalfBytes;
      if (draft && p.prefix_grouped) {
        // Grouped layout: box = lane -> (tensor K/V = lane & 1, 8-slot group lane >> 1), both halves
        // (3-D map {64 dims, rows, 2 halves}).
        const int nbox = (nkeys + kDraftBoxRows - 1) / kDraftBoxRows;
        if (lane == 0) mbar_arrive_expect_tx(full_bar, 2u * nbox * kGroupBytes);
        const int ib = lane >> 1;
        if (ib < nbox) {
          const int y0 = (cu.c * p.hkv + h) * p.n_max + key0;
          tma_load_3d(kdst + kv * kKVTileBytes + ib * kGroupBytes, kv ? &maps.dv : &maps.dk, 0,
                      y0 + ib * kDraftBoxRows, 0, full_bar, policy);
        }
      } else if (draft) {
        const int nbox = (nkeys + kDraftBoxRows - 1) / kDraftBoxRows;
        if (lane == 0) mbar_arrive_expect_tx(full_bar, nbox * kDraftBoxRows * 128 * 4);
        if (i < nbox) {
          const int y0 = (cu.c * p.hkv + h) * p.n_max + key0;
          tma_load_2d(dst + i * kDraftBoxRows * 128, kv ? &maps.dv : &maps.dk, hf * 64, y0 + i * kDraftBoxRows,
                      full_bar, policy);
        }
      } else if (p.paged && p.prefix_grouped) {
        // Grouped layout (bf16): box = lane -> (tensor K/V = lane & 1, box lane >> 1), a box of whole
        // 8-key groups with both 64-dim halves: one page of P < 64 tokens, or the tile's 64-token
        // slice of a larger page.  Half the boxes of the halves layout, each twice the bytes.
        const int P = p.page_size;
        const bool small_pages = P < kTileKeys;
        const int nbox = small_pages ? (nkeys + P - 1) / P : 1;
        const uint32_t box_bytes = small_pages ? static_cast<uint32_t>(P) * 256u : static_cast<uint32_t>(kKVTileBytes);
        if (lane == 0) mbar_arrive_expect_tx(full_bar, 2u * nbox * box_bytes);
        const int ib = lane >> 1;
        if (ib < nbox) {
          int pid = pids[0];
#pragma unroll
          for (int k = 1; k < kTileKeys / 8; ++k)
            if (ib == k) pid = pids[k];
          const int y = ((pid * p.hkv + h) * P + (small_pages ? 0 : key0 % P)) >> 3;
          tma_load_4d_hint(kdst + kv * kKVTileBytes + ib * box_bytes, kv ? &maps.tv : &maps.tk, 0, 0, 0, y,
                           full_bar, policy);
        }
      } else if (p.paged) {
        // bf16: boxes of 64 dims per half; fp8 (p.fp8): one box of whole 128-byte rows, into the
        // upper half of the tile (the lanes of half 1 skip), decoded from there by the consumers.
        const int br = p.box_rows;
        const int nbox = (nkeys + br - 1) / br;
        if (lane == 0) mbar_arrive_expect_tx(full_bar, nbox * br * 128 * (p.fp8 ? 2 : 4));
        if (i < nbox && !(p.fp8 && hf)) {
          int pid = pids[0];
#pragma unroll
          for (int k = 1; k < kTileKeys / 8; ++k)
            if (i == k) pid = pids[k];
          const int krow = key0 + i * br;
          const int y = (pid * p.hkv + h) * p.page_size + (krow % p.page_size);
          const uint32_t d0 = p.fp8 ? kdst + kv * kKVTileBytes + kHalfBytes : dst;
          tma_load_2d(d0 + i * br * 128, kv ? &maps.tv : &maps.tk, p.fp8 ? 0 : hf * 64, y, full_bar, policy);
        }
      } else {
        if (lane == 0) mbar_arrive_expect_tx(full_bar, kTileKeys * 128 * (p.fp8 ? 2 : 4));
        if (i == 0 && !(p.fp8 && hf)) {
          const int y = (cu.c * p.hkv + h) * p.l_cap + key0;
          const uint32_t d0 = p.fp8 ? kdst + kv * kKVTileBytes + kHalfBytes : dst;
          tma_load_2d(d0, kv ? &maps.tv : &maps.tk, p.fp8 ? 0 : hf * 64, y, full_bar, policy);
        }
      }
    }
    ++issued;
    cursor_next(cu, p, s_len);
    if (++stage == pipe.stages) {
      stage = 0;
      phase ^= 1u;
    }
  }
  if (lane == 0) *pipe.issued = issued;
}

// After the roles finish: if a wait timed out, wait (bounded) for every TMA
// load still in flight so no copy lands in shared memory after the CTA exits.
// Called by one thread after a block-wide barrier.
__device__ __forceinline__ void drain_after_abort(const AttnParams& p, const Pipe& pipe, int consumed) {
  if (!*pipe.abort) return;
  for (int k = consumed; k < *pipe.issued; ++k) {
    const int st = k % pipe.stages;
    const uint32_t par = static_cast<uint32_t>((k / pipe.stages) & 1);
    if (!mbar_wait(smem_addr(&pipe.full[st]), par, p.err)) break;
  }
}

}  // namespace
}  // namespace dev
}  // namespace kvshot
