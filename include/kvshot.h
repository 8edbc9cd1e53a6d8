/*
 * kvshot.h -- C ABI of libkvshot, GB300 (sm_103a) draft attention for
 * KV-reuse speculative drafting.
 *
 * The drafter of a KV-reuse speculative decoder re-attends, with its own
 * query, to the target model's key/value cache instead of (or next to) the
 * target's hidden state: a' = sum_i alpha_i(q') v_i with
 * alpha_i(q') = softmax_i(q'^T k_i)  (arXiv 2604.26412, Sec. 2.2,
 * Eq. "kv-reattention").  Its memory M_i holds the target K/V of the verified
 * prefix (j <= t) followed by K/V the drafter produced for its own earlier
 * draft positions (j > t)  (Sec. 3.4, Eq. "cross-attn"; App. B,
 * "Cross-attention memory").  The same attention step serves the KV-only
 * drafter (Sec. 3.2) and the cross-attention branch o_i of the hybrid
 * gated-delta drafter (Sec. 3.4).  Draft positions form a chain (K draft
 * tokens drafted one after another, Sec. 4.2) or a tree (tree verification
 * with a (8, 10, 60) draft tree, Sec. 3.1 and 3.5); a draft node sees every
 * verified prefix token plus itself and its ancestors among the draft nodes.
 *
 * Conventions for every entry point:
 *  - All tensor pointers are DEVICE pointers owned by the caller.  The
 *    library never allocates; scratch space is the caller's workspace.
 *  - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream).  Nothing synchronises the host.
 *  - Argument errors are found on the host, before anything is enqueued, and
 *    returned as a kvshot_status; nothing is launched then.
 *  - Errors only visible on the device (a page id outside the pool, a
 *    sequence length above the stated bound, a parent index that is not an
 *    earlier node, a pipeline wait that timed out) are recorded in
 *    desc->err_flag (if non-NULL): the first error code is stored with an
 *    atomic compare-and-swap from 0.  Outputs of the affected call are then
 *    unspecified.  No kernel traps.
 *  - bf16 tensors are row-major with the innermost dimension head_dim (= 128).
 */
#ifndef KVSHOT_H
#define KVSHOT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* kvshot_stream_t; /* same handle type as cudaStream_t */

typedef enum kvshot_status {
  KVSHOT_OK = 0,
  KVSHOT_ERR_NULL = 1,          /* a required pointer is NULL */
  KVSHOT_ERR_SHAPE = 2,         /* inconsistent or out-of-range sizes in the descriptor */
  KVSHOT_ERR_ALIGN = 3,         /* a pointer is not aligned as stated below */
  KVSHOT_ERR_UNSUPPORTED = 4,   /* valid but outside this build (head_dim != 128, tree with > 64 nodes, ...) */
  KVSHOT_ERR_TREE = 5,          /* (device) tree_parent[i] is not in [-1, i) */
  KVSHOT_ERR_WORKSPACE = 6,     /* workspace missing, misaligned or smaller than the size query returns */
  KVSHOT_ERR_CUDA = 7,          /* a CUDA runtime/driver call failed (tensor map encode, launch) */
  KVSHOT_ERR_DEVICE_BOUNDS = 8, /* (device) page id outside the pool or seq_len above its bound */
  KVSHOT_ERR_TIMEOUT = 9        /* (device) a pipeline wait gave up after its time limit */
} kvshot_status;

/* desc->flags */
#define KVSHOT_TREE 0x1u       /* draft nodes form a tree given by tree_parent (else a chain) */
#define KVSHOT_FORCE_CC 0x2u   /* use the CUDA-core kernel whatever the row count (measurement aid) */
#define KVSHOT_FORCE_MMA 0x4u  /* use the mma.sync tensor-core kernel whatever the row count (measurement aid) */
#define KVSHOT_FORCE_TC 0x8u   /* use the tcgen05 / tensor-memory kernel (needs 128 % (hq / hkv) == 0) */
/* Let the attention kernel start while the kernel enqueued just before the call is still running
 * (programmatic dependent launch): it then reads seq_lens, page_table, target_k/v and tree_parent,
 * and starts the first target K/V loads, before that kernel has finished, and waits for it only
 * before it reads q or draft_k/v or writes anything.  Set it only when the preceding kernel does
 * not write seq_lens, page_table, target_k, target_v or tree_parent (kvshot_draft_append, which
 * writes q and the draft K/V, qualifies). */
#define KVSHOT_OVERLAP_PREVIOUS 0x10u
/* The target cache (target_k, target_v) holds fp8 E4M3 codes (OCP FP8: 1 sign bit, 4 exponent
 * bits with bias 7, 3 mantissa bits, subnormals, codes 0x7F and 0xFF NaN, no infinities), one byte
 * per element in the same row layout as the bf16 cache ([..][128] per token and KV head).  The
 * key and value of a target token are decoded as
 *   k = e4m3(code) * 2^desc->k_scale_exp,   v = e4m3(code) * 2^desc->v_scale_exp
 * which is exact in bf16 for |exponent| <= 64; attention then proceeds as for a bf16 cache.  The
 * draft K/V stay bf16.  Both tensor-core kernels then multiply in f16 (e4m3 -> f16 is exact; q,
 * P and the draft K/V are rounded to f16, which keeps more mantissa than bf16; only magnitudes below
 * 2^-14 lose bits).  Stacks of 17 to 128 rows run on the tcgen05 kernel, which decodes the codes
 * into f16 tiles in shared memory; the others on the m16n8k16 kernel, which decodes them in
 * registers.  KVSHOT_FORCE_TC with more than 128 rows and KVSHOT_FORCE_CC return
 * KVSHOT_ERR_UNSUPPORTED.  Not in the paper: a cache-compression variant that halves the bytes the
 * kernel reads per target token. */
#define KVSHOT_TARGET_FP8 0x20u

/*
 * Problem descriptor shared by kvshot_draft_attn and kvshot_draft_append.
 *
 * A "cache" is one independent KV cache: one sequence when one target layer
 * is reused, or one (sequence, reused target layer) pair when several target
 * layers are attended separately (KV-only head concatenation, Sec. 3.2).
 * Caches of one sequence are consecutive and share that sequence's draft tree.
 */
typedef struct kvshot_attn_desc {
  int32_t num_caches;        /* C >= 1 (<= 1024) */
  int32_t num_seqs;          /* B >= 1, C % B == 0; cache c belongs to sequence c / (C / B) */
  int32_t hq;                /* query heads */
  int32_t hkv;               /* KV heads; hq % hkv == 0 (GQA group G = hq / hkv) */
  int32_t head_dim;          /* must be 128 */
  int32_t page_size;         /* paged layout: tokens per page: 8, 16, 32, 64, 128, 192 or 256 */
  int32_t max_pages_per_seq; /* paged layout: row stride of page_table */
  int32_t num_pages;         /* paged layout: pages in the target_k / target_v pools */
  int32_t l_cap;             /* contiguous layout: token capacity per (cache, KV head) */
  int32_t max_seq_len;       /* host-known upper bound on every seq_lens[c]; sizes the work plan */
  int32_t n_nodes;           /* N: draft nodes present; draft slots 0..N-1 hold their K/V */
  int32_t n_query;           /* Nq: the last Nq draft nodes are the query rows (Nq <= N) */
  int32_t n_max;             /* draft buffer capacity in slots (N <= n_max) */
  float scale;               /* softmax scale on q.k, > 0; 0 selects 1/sqrt(head_dim); negative -> KVSHOT_ERR_SHAPE */
  uint32_t flags;            /* KVSHOT_TREE, at most one of KVSHOT_FORCE_CC / _MMA / _TC */
  int32_t num_ctas;          /* persistent CTAs to launch; 0 = one full wave on this GPU */
  void* workspace;           /* device scratch, 256-byte aligned; see kvshot_draft_attn_workspace_size */
  size_t workspace_bytes;
  int32_t* err_flag;         /* optional device int32, 0 before the call; see conventions above */
  int32_t k_scale_exp;       /* KVSHOT_TARGET_FP8: target keys are e4m3 x 2^k_scale_exp, |exp| <= 64 */
  int32_t v_scale_exp;       /* KVSHOT_TARGET_FP8: target values are e4m3 x 2^v_scale_exp, |exp| <= 64 */
  uint32_t wait_limit_ns;    /* watchdog: longest any one wait of the attention kernels' load/compute
                                pipeline may take, in ns; 0 = 2 s.  A wait that runs past it records
                                KVSHOT_ERR_TIMEOUT; the kernel then stops computing, waits (2 s at most
                                each) for the copies and tensor-core operations it already issued, and
                                returns, leaving the outputs unspecified.  Setting it near zero makes every
                                CTA give up on its first unfinished wait: a way to exercise that path. */
} kvshot_attn_desc;

/*
 * Bytes of workspace kvshot_draft_attn needs for `desc` on the current device
 * (partial softmax states of work pieces that straddle CTAs).  Returns 0 if the descriptor is invalid.  The size depends on the
 * shape fields, flags, num_ctas and the device's SM count, not on pointers.
 */
size_t kvshot_draft_attn_workspace_size(const kvshot_attn_desc* desc);

/*
 * Draft attention.  For every cache c, query row n_local in [0, Nq) (draft
 * node n = N - Nq + n_local) and query head h (KV head h / G):
 *
 *   keys  = { prefix tokens j in [0, L_c) }  U  { draft slots m : m == n or m is an ancestor of n }
 *   s_k   = scale * q . k_k
 *   lse   = log sum_k exp(s_k)                          (natural log)
 *   out   = sum_k exp(s_k - lse) v_k                    (fp32 accumulate, rounded to bf16)
 *
 * where L_c = seq_lens[c] (Sec. 2.2 Eq. "kv-reattention" over M_i of Sec. 3.4 / App. B).
 * A chain (flags without KVSHOT_TREE) means node n's ancestors are 0..n-1.
 *
 * q:           [C, Nq, hq, 128] bf16, 16-byte aligned.
 * target_k/v:  paged (page_table != NULL): [num_pages, hkv, page_size, 128] bf16;
 *              contiguous (page_table == NULL): [C, hkv, l_cap, 128] bf16.  16-byte aligned.
 *              Rows past L_c may hold anything (NaN included); they are never used.
 * page_table:  [C, max_pages_per_seq] int32; entry p of cache c is the pool page of tokens
 *              [p * page_size, (p + 1) * page_size).  Only the first ceil(L_c / page_size) entries are read.
 * seq_lens:    [C] int32, 0 <= L_c <= min(max_seq_len, capacity).
 * draft_k/v:   [C, hkv, n_max, 128] bf16, 16-byte aligned; slots 0..N-1 are read.
 * tree_parent: [B, N] int32, parent[i] in [-1, i) (-1 = child of the last verified token);
 *              read only with KVSHOT_TREE (then N <= 64).  May be NULL for a chain.
 * out:         [C, Nq, hq, 128] bf16, 16-byte aligned, must not alias any input.
 * lse:         [C, Nq, hq] fp32 (natural log), 4-byte aligned.
 * Nq == 0 is a no-op returning KVSHOT_OK.
 */
kvshot_status kvshot_draft_attn(const kvshot_attn_desc* desc, const void* q, const void* target_k,
                                const void* target_v, const int32_t* page_table, const int32_t* seq_lens,
                                const void* draft_k, const void* draft_v, const int32_t* tree_parent,
                                void* out, float* lse, kvshot_stream_t stream);

/* Bytes of device scratch built into the library for kvshot_draft_attn_static (64 MiB: enough for the
 * plan of a 64-node whole tree over 16 caches x 8 KV heads, 256 stacked rows per head, ~34 MB). */
#define KVSHOT_STATIC_WORKSPACE_BYTES (64u * 1024u * 1024u)

/*
 * kvshot_draft_attn_static -- the same computation, arguments and results as
 * kvshot_draft_attn, for callers that cannot allocate device memory: code
 * handed only device pointers by a host framework that owns all allocation,
 * a serving loop whose memory pool is fully reserved up front, or a hot path
 * that must not call cudaMalloc (which can synchronise the device and stall
 * every other stream).  The paper has no counterpart; this is an interface
 * convenience only.
 *
 * Instead of desc->workspace (ignored, as is desc->workspace_bytes) the call
 * uses a fixed scratch array of KVSHOT_STATIC_WORKSPACE_BYTES inside the
 * library; every GPU that loads the library holds that array until the
 * process exits.  The call itself allocates nothing.
 *  - Descriptors whose work plan needs more scratch than that
 *    (kvshot_draft_attn_workspace_size(desc) > KVSHOT_STATIC_WORKSPACE_BYTES)
 *    are rejected with KVSHOT_ERR_WORKSPACE before anything is launched.
 *  - The first call on each device looks up the array's device address (with
 *    that device current) and keeps it for the life of the process; make that
 *    first call before any stream capture.  The kept address belongs to the
 *    device's primary context: after cudaDeviceReset (or any teardown of that
 *    context) it is stale, and the entry point must not be called again in
 *    that process.
 *  - All calls on a device share the one array and it keeps the last call's
 *    contents.  Nothing in it has to start at zero, but two calls whose
 *    kernels overlap on the GPU (e.g. on different streams without ordering)
 *    race on it and corrupt each other's results; keep such calls ordered.
 */
kvshot_status kvshot_draft_attn_static(const kvshot_attn_desc* desc, const void* q, const void* target_k,
                                       const void* target_v, const int32_t* page_table, const int32_t* seq_lens,
                                       const void* draft_k, const void* draft_v, const int32_t* tree_parent,
                                       void* out, float* lse, kvshot_stream_t stream);

/*
 * Draft append with RoPE: the drafter's new K/V for draft positions j > t
 * enter M_i (App. B: past the verified prefix the memory holds keys and
 * values that the drafter computes itself with its own projection weights;
 * those projections are upstream GEMMs), with rotary position embedding
 * applied to q and k (RoPE re-application, Sec. 3.2).
 *
 * For cache c and new node i in [0, n_new) at position pos = positions[c, i]:
 *   theta_j = pos * rope_base^(-2j / 128),  j in [0, 64)
 *   rot(x)[j]      = x[j] cos(theta_j) - x[j + 64] sin(theta_j)
 *   rot(x)[j + 64] = x[j + 64] cos(theta_j) + x[j] sin(theta_j)
 *   q_out[c, i, h]              = bf16(rot(q_in[c, i, h]))      for h < hq
 *   draft_k[c, kh, n0 + i]      = bf16(rot(k_in[c, i, kh]))     for kh < hkv
 *   draft_v[c, kh, n0 + i]      = v_in[c, i, kh]                (copied bit for bit)
 * Angles and rotations are computed in fp64 and rounded once to bf16 (nearest even).
 *
 * q_in:  [C, n_new, hq, 128] bf16; k_in, v_in: [C, n_new, hkv, 128] bf16; positions: [C, n_new] int32 >= 0.
 * draft_k/v: [C, hkv, n_max, 128] bf16 (desc->n_max); requires 0 <= n0 and n0 + n_new <= n_max.
 * q_out: [C, n_new, hq, 128] bf16; may equal q_in (in place) but must not partially overlap it.
 * All bf16 pointers 16-byte aligned.  Only num_caches, hq, hkv, head_dim and n_max of desc are read.
 * n_new == 0 is a no-op returning KVSHOT_OK.
 */
kvshot_status kvshot_draft_append(const kvshot_attn_desc* desc, const void* q_in, const void* k_in,
                                  const void* v_in, const int32_t* positions, int32_t n0, int32_t n_new,
                                  float rope_base, void* draft_k, void* draft_v, void* q_out,
                                  kvshot_stream_t stream);

/*
 * Gated-delta fusion of the hybrid drafter (Sec. 3.4, Eqs. "self-attn",
 * "cross-attn", "delta" and "fusion").  For every draft token t, with n_t the
 * self-attention branch (the EAGLE-3 path) and o_t the cross-attention
 * branch (re-attention to the target KV):
 *   delta_t = o_t - n_t
 *   g_t     = sigmoid(W_g [n_t; o_t; delta_t] + b_g)
 *   h_t     = n_t + g_t (.) (W_delta delta_t)
 * The attention of both branches is kvshot_draft_attn: over the target prefix
 * and the draft KV for o, over the drafter's own draft KV alone (every
 * seq_lens[c] = 0) for n.  Products accumulate in fp32 and delta is never
 * rounded (W delta is formed as W o - W n in fp32); h is rounded once to bf16
 * (nearest even).
 *
 * n, o:     [T, d] bf16, row-major (token-major), 16-byte aligned.
 * w_g:      [d, 3d] bf16, row-major: row i holds output feature i's weights
 *           over the inputs [n; o; delta].  16-byte aligned.
 * b_g:      [d] bf16, 8-byte aligned.
 * w_delta:  [d, d] bf16, row-major, 16-byte aligned.
 * h:        [T, d] bf16, 8-byte aligned; must not overlap n, o or the workspace.
 * desc->hidden = d: a positive multiple of 128, at most 32768 (else
 * KVSHOT_ERR_UNSUPPORTED); desc->num_tokens = T >= 0 (0: no-op), T * d < 2^31.
 * Workspace: kvshot_gated_delta_workspace_size(desc) bytes (the fp32 partial
 * products, 16 T d bytes), 256-byte aligned; nothing in it has to be
 * initialised.  Errors follow the conventions at the top of this file.
 */
typedef struct kvshot_fusion_desc {
  int32_t num_tokens;        /* T */
  int32_t hidden;            /* d */
  void* workspace;           /* device scratch, 256-byte aligned */
  size_t workspace_bytes;
  int32_t* err_flag;         /* optional device int32, 0 before the call (KVSHOT_ERR_TIMEOUT) */
} kvshot_fusion_desc;

/* Bytes of workspace kvshot_gated_delta needs; 0 if the descriptor is invalid. */
size_t kvshot_gated_delta_workspace_size(const kvshot_fusion_desc* desc);

kvshot_status kvshot_gated_delta(const kvshot_fusion_desc* desc, const void* n, const void* o, const void* w_g,
                                 const void* b_g, const void* w_delta, void* h, kvshot_stream_t stream);

/*
 * Linear projection of multi-layer target KV for the KV-only drafter
 * (Sec. 3.2, injection strategy "linear projection"; "Proj + RoPE fix").
 * For every newly verified token t (desc->num_tokens = T of them), with
 * d_kv = hkv * 128 and L = desc->num_layers sampled target layers:
 *   K'(t) = W_K [K_1(t); ...; K_L(t)],   V'(t) = W_V [V_1(t); ...; V_L(t)]
 * and, with KVSHOT_PROJECT_ROPE, K'(t) is rotated again by RoPE at the
 * token's position (rotate-half pairs (j, j + 64) of every head,
 * theta_j = pos * rope_base^(-2j/128), as in kvshot_draft_append).  K'(t) and
 * V'(t) are rounded to bf16 and stored in slot positions[t] of cache
 * token_cache[t] of the reused cache that kvshot_draft_attn reads as its
 * target K/V; other slots are left untouched.  Products accumulate in fp32.
 *
 * k_in, v_in:  [T, L, hkv, 128] bf16: the tokens' K / V of the L layers (K post-RoPE, as cached).
 * w_k, w_v:    [d_kv, L * d_kv] bf16, row-major (row i: output feature i over the concatenated inputs).
 * token_cache: [T] int32 in [0, num_caches); positions: [T] int32 >= 0, below the cache's capacity.
 * page_table:  paged cache (non-NULL): [num_caches, max_pages_per_seq] int32; k_out / v_out are
 *              [num_pages, hkv, page_size, 128] bf16.  Contiguous (NULL): k_out / v_out are
 *              [num_caches, hkv, l_cap, 128] bf16.
 * All bf16 pointers 16-byte aligned, int32 pointers 4-byte aligned.  num_layers <= 8, hkv <= 64.
 * Device-side errors (a cache, position or page id out of range) skip that token's store and set
 * KVSHOT_ERR_DEVICE_BOUNDS.  T == 0 is a no-op.
 * Workspace: kvshot_kv_project_workspace_size(desc) bytes (fp32 partial products, 8 L T d_kv bytes), 256-byte aligned,
 * no initialisation needed.
 */
#define KVSHOT_PROJECT_ROPE 0x1u /* re-apply RoPE to the projected keys ("Proj + RoPE fix") */

typedef struct kvshot_project_desc {
  int32_t num_tokens;        /* T */
  int32_t num_layers;        /* L >= 1 */
  int32_t hkv;               /* KV heads */
  int32_t head_dim;          /* must be 128 */
  int32_t num_caches;        /* caches of the output (reused) cache */
  int32_t page_size;         /* paged output: tokens per page */
  int32_t max_pages_per_seq; /* paged output: row stride of page_table */
  int32_t num_pages;         /* paged output: pages in the pools */
  int32_t l_cap;             /* contiguous output: token capacity per (cache, KV head) */
  float rope_base;           /* > 0 (used with KVSHOT_PROJECT_ROPE) */
  uint32_t flags;            /* KVSHOT_PROJECT_ROPE or 0 */
  void* workspace;           /* device scratch, 256-byte aligned */
  size_t workspace_bytes;
  int32_t* err_flag;         /* optional device int32, 0 before the call */
} kvshot_project_desc;

/* Bytes of workspace kvshot_kv_project needs (0 if the descriptor is invalid; the layout is read
 * from page_size > 0 for this query). */
size_t kvshot_kv_project_workspace_size(const kvshot_project_desc* desc);

kvshot_status kvshot_kv_project(const kvshot_project_desc* desc, const void* k_in, const void* v_in,
                                const void* w_k, const void* w_v, const int32_t* token_cache,
                                const int32_t* positions, const int32_t* page_table, void* k_out, void* v_out,
                                kvshot_stream_t stream);

/*
 * kvshot_draft_append with QK-norm (App. D, Tab. ablations, the "QK-Norm"
 * training regime, which the paper names without a formula; read as Qwen3's
 * attention, which normalises q and k per head before RoPE): every
 * 128-wide q and k head is first scaled to unit RMS and by its weights,
 *   x <- x / sqrt(mean_j x_j^2 + eps) * w        (w = q_norm_w or k_norm_w)
 * and then rotated exactly as kvshot_draft_append does; v is stored as is.
 * Computed in fp32 and rounded once to bf16 (so not bit-identical to an fp64
 * evaluation: the results are within one bf16 rounding step of it).
 * q_norm_w, k_norm_w: [128] bf16, 4-byte aligned.  eps > 0 (Qwen3: 1e-6).
 * Every other argument as for kvshot_draft_append.
 */
kvshot_status kvshot_draft_append_qknorm(const kvshot_attn_desc* desc, const void* q_in, const void* k_in,
                                         const void* v_in, const int32_t* positions, int32_t n0, int32_t n_new,
                                         float rope_base, const void* q_norm_w, const void* k_norm_w, float eps,
                                         void* draft_k, void* draft_v, void* q_out, kvshot_stream_t stream);

/* Static description of a status code (never NULL). */
const char* kvshot_status_string(kvshot_status status);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t kvshot_version(void);

#ifdef __cplusplus
}
#endif
#endif /* KVSHOT_H */
