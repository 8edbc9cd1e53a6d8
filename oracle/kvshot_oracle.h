/*
 * kvshot_oracle.h -- CPU fp64 oracle for KV-reuse draft attention.
 *
 * TEST INFRASTRUCTURE ONLY.  This is the plain, slow, obviously-correct
 * definition that the CUDA library is checked against.  Only the test suite,
 * the package's smoke() self-check and the benchmark's CPU-baseline leg may
 * load it.  It shares no code, header, table or helper with the CUDA library
 * (paper_2604_26412_gb300/csrc, include/kvshot.h) and it never includes them.
 *
 * What it computes (the paper's notation):
 *   - re-attention of a draft query q' over target key/value pairs,
 *     a' = sum_i alpha_i(q') v_i with alpha = softmax(q'^T k_i)
 *     (Sec. 2.2, Eq. "kv-reattention"), with the usual 1/sqrt(d) scale;
 *   - the cross-attention memory M_i of the hybrid drafter (Sec. 3.4,
 *     Eq. "cross-attn"; App. B "Cross-attention memory"): verified prefix
 *     tokens j <= t take the target model's K/V, later positions j > t take
 *     the drafter's own K/V;
 *   - over a draft chain (autoregressive drafting) or a draft tree (tree
 *     verification, Sec. 3.5): a draft node sees exactly itself and its
 *     ancestors among the draft nodes, and every verified prefix token;
 *   - RoPE (rotate-half) applied to newly drafted q and k before they are
 *     appended to the draft KV (Sec. 3.2 re-applies RoPE to reused KV).
 *
 * All bf16 inputs are passed as raw uint16 bit patterns and widened exactly.
 * Accumulation is fp64.  Return value: 0 on success, a positive error code on
 * invalid input (see KVO_ERR_*); nothing is written on error.
 */
#ifndef KVSHOT_ORACLE_H
#define KVSHOT_ORACLE_H
#include <stdint.h>
#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  KVO_OK = 0,
  KVO_ERR_SHAPE = 2,     /* inconsistent sizes */
  KVO_ERR_TREE = 5,      /* tree_parent[i] not in [-1, i) */
  KVO_ERR_PAGE = 8,      /* page id outside the pool, or seq_len above capacity */
};

typedef struct kvo_desc {
  int32_t num_caches;        /* C: independent KV caches (sequences x reused target layers) */
  int32_t num_seqs;          /* B: sequences; cache c belongs to sequence c / (C / B) */
  int32_t hq, hkv, head_dim; /* query heads, KV heads (hq % hkv == 0), head dimension */
  int32_t paged;             /* 1: target K/V in pages [num_pages, hkv, page_size, D]; 0: [C, hkv, l_cap, D] */
  int32_t page_size, max_pages_per_seq, num_pages;
  int32_t l_cap;
  int32_t n_nodes;           /* N: draft nodes present; draft slots 0..N-1 hold their K/V */
  int32_t n_query;           /* Nq: the last Nq draft nodes are the query rows */
  int32_t n_max;             /* draft buffer capacity: draft K/V are [C, hkv, n_max, D] */
  int32_t tree;              /* 0: chain (node n's ancestors are 0..n-1); 1: tree_parent decides */
  double scale;              /* softmax scale; 0 selects 1/sqrt(head_dim) */
} kvo_desc;

/* Masked GQA attention over [target prefix | draft KV].
 * q:   [C, Nq, hq, D] bf16 bits.  Query row n_local is draft node N - Nq + n_local.
 * tk, tv: target K/V (paged or contiguous, see kvo_desc).  page_table: [C, max_pages_per_seq].
 * seq_lens: [C] verified prefix length L_c.
 * dk, dv: draft K/V [C, hkv, n_max, D] bf16 bits.
 * tree_parent: [B, N] (ignored for a chain; may be NULL then).
 * out: [C, Nq, hq, D] fp64.  lse: [C, Nq, hq] fp64, natural log of sum exp(scale q.k).
 * nthreads: worker threads (0 = all hardware threads). */
int kvo_attn(const kvo_desc* d, const uint16_t* q, const uint16_t* tk, const uint16_t* tv,
             const int32_t* page_table, const int32_t* seq_lens, const uint16_t* dk,
             const uint16_t* dv, const int32_t* tree_parent, double* out, double* lse,
             int nthreads);

/* Softmax probabilities of one query row over its key list, for tests.
 * Writes probs[0 .. L_c + N): entries 0..L_c-1 are the prefix keys, entries L_c + m are
 * draft slot m (exactly 0 for draft slots the row cannot see). */
int kvo_attn_probs(const kvo_desc* d, const uint16_t* q, const uint16_t* tk,
                   const int32_t* page_table, const int32_t* seq_lens, const uint16_t* dk,
                   const int32_t* tree_parent, int32_t c, int32_t n_local, int32_t h,
                   double* probs);

/* Draft append: RoPE (rotate-half, theta_j = pos * base^(-2j/D)) on new q and k,
 * then k, v stored into draft slots n0 .. n0+n_new-1.
 * q_in: [C, n_new, hq, D], k_in/v_in: [C, n_new, hkv, D], positions: [C, n_new].
 * draft_k/draft_v: [C, hkv, n_max, D] (updated in place), q_out: [C, n_new, hq, D].
 * bf16 outputs are fp64 results rounded to nearest-even.  q_rot_f64 / k_rot_f64
 * (optional) receive the unrounded rotated values in the q_in / k_in layouts. */
int kvo_append(const kvo_desc* d, const uint16_t* q_in, const uint16_t* k_in, const uint16_t* v_in,
               const int32_t* positions, int32_t n0, int32_t n_new, double rope_base,
               uint16_t* draft_k, uint16_t* draft_v, uint16_t* q_out,
               double* q_rot_f64, double* k_rot_f64);

/* fp64 -> bf16 bits, round to nearest, ties to even (exposed for tests). */
uint16_t kvo_round_bf16(double x);

#ifdef __cplusplus
}
#endif
#endif
