/*
 * kvshot_oracle.cpp -- CPU fp64 oracle for KV-reuse draft attention.
 *
 * TEST INFRASTRUCTURE ONLY (see kvshot_oracle.h).  Plain loops, fp64
 * accumulation, one std::thread pool over (cache, query head).  No blocking,
 * no online softmax, no split/merge: every query row's full key list is
 * materialised and the softmax is taken directly from its definition.
 *
 * Definitions followed:
 *   attention:  Sec. 2.2, Eq. "kv-reattention": a' = sum_i alpha_i(q') v_i,
 *               alpha_i = exp(q'.k_i) / sum_j exp(q'.k_j), scores scaled by
 *               1/sqrt(d) (standard transformer practice; the paper's equation
 *               omits the scale, so it is a parameter here).
 *   memory M_i: Sec. 3.4 Eq. "cross-attn" and App. B: verified prefix tokens
 *               (target K/V) followed by the drafter's own K/V.
 *   draft mask: a chain node n sees draft slots 0..n; a tree node sees itself
 *               and its ancestors (tree verification, Sec. 3.5).
 *   RoPE:       rotate-half pairs (j, j + D/2), theta_j = pos * base^(-2j/D),
 *               re-applied to drafted keys (Sec. 3.2 "Proj + RoPE fix").
 */
#include "kvshot_oracle.h"

#include <atomic>
#include <cfenv>
#include <cmath>
#include <cstring>
#include <thread>
#include <vector>

namespace {

double widen_bf16(uint16_t h) {
  uint32_t u = static_cast<uint32_t>(h) << 16;
  float f;
  std::memcpy(&f, &u, sizeof f);
  return static_cast<double>(f);
}

int check_desc(const kvo_desc* d) {
  if (d->num_caches <= 0 || d->num_seqs <= 0 || d->num_caches % d->num_seqs) return KVO_ERR_SHAPE;
  if (d->hq <= 0 || d->hkv <= 0 || d->hq % d->hkv || d->head_dim <= 0 || d->head_dim % 2) return KVO_ERR_SHAPE;
  if (d->n_nodes < 0 || d->n_query < 0 || d->n_query > d->n_nodes || d->n_nodes > d->n_max) return KVO_ERR_SHAPE;
  if (d->paged) {
    if (d->page_size <= 0 || d->max_pages_per_seq < 0 || d->num_pages < 0) return KVO_ERR_SHAPE;
  } else if (d->l_cap < 0) {
    return KVO_ERR_SHAPE;
  }
  return KVO_OK;
}

int prefix_capacity(const kvo_desc* d) {
  return d->paged ? d->page_size * d->max_pages_per_seq : d->l_cap;
}

// Row of the target cache holding prefix token j of cache c, KV head h.
const uint16_t* target_row(const kvo_desc* d, const uint16_t* base, const int32_t* page_table,
                           int c, int h, int j) {
  size_t row;
  if (d->paged) {
    int page = page_table[static_cast<size_t>(c) * d->max_pages_per_seq + j / d->page_size];
    row = (static_cast<size_t>(page) * d->hkv + h) * d->page_size + j % d->page_size;
  } else {
    row = (static_cast<size_t>(c) * d->hkv + h) * d->l_cap + j;
  }
  return base + row * d->head_dim;
}

const uint16_t* draft_row(const kvo_desc* d, const uint16_t* base, int c, int h, int m) {
  size_t row = (static_cast<size_t>(c) * d->hkv + h) * d->n_max + m;
  return base + row * d->head_dim;
}

// visible[m] = 1 iff draft slot m is node n itself or one of its ancestors.
void draft_visibility(const kvo_desc* d, const int32_t* parents_of_seq, int n,
                      std::vector<char>& visible) {
  visible.assign(d->n_nodes, 0);
  if (!d->tree) {
    for (int m = 0; m <= n; ++m) visible[m] = 1;
    return;
  }
  for (int m = n; m >= 0; m = parents_of_seq[m]) visible[m] = 1;
}

int validate_contents(const kvo_desc* d, const int32_t* page_table, const int32_t* seq_lens,
                      const int32_t* tree_parent) {
  const int cap = prefix_capacity(d);
  for (int c = 0; c < d->num_caches; ++c) {
    int L = seq_lens[c];
    if (L < 0 || L > cap) return KVO_ERR_PAGE;
    if (d->paged) {
      for (int p = 0; p < (L + d->page_size - 1) / d->page_size; ++p) {
        int page = page_table[static_cast<size_t>(c) * d->max_pages_per_seq + p];
        if (page < 0 || page >= d->num_pages) return KVO_ERR_PAGE;
      }
    }
  }
  if (d->tree) {
    for (int b = 0; b < d->num_seqs; ++b)
      for (int i = 0; i < d->n_nodes; ++i) {
        int p = tree_parent[static_cast<size_t>(b) * d->n_nodes + i];
        if (p < -1 || p >= i) return KVO_ERR_TREE;
      }
  }
  return KVO_OK;
}

struct RowInputs {
  const kvo_desc* d;
  const uint16_t *q, *tk, *tv, *dk, *dv;
  const int32_t *page_table, *seq_lens, *tree_parent;
};

// Scores s_j = scale * q.k_j over the row's visible keys (prefix first, then
// visible draft slots).  Fills key_rows (pointers into K and V) for the caller.
void row_scores(const RowInputs& in, int c, int n_local, int h, std::vector<double>& s,
                std::vector<const uint16_t*>& vrows, std::vector<int>& key_ids) {
  const kvo_desc* d = in.d;
  const int D = d->head_dim;
  const int G = d->hq / d->hkv;
  const int kvh = h / G;
  const int n = d->n_nodes - d->n_query + n_local;
  const int L = in.seq_lens[c];
  const int seq = c / (d->num_caches / d->num_seqs);
  const double scale = d->scale != 0.0 ? d->scale : 1.0 / std::sqrt(static_cast<double>(D));
  const uint16_t* qrow = in.q + ((static_cast<size_t>(c) * d->n_query + n_local) * d->hq + h) * D;

  std::vector<char> visible;
  draft_visibility(d, in.tree_parent ? in.tree_parent + static_cast<size_t>(seq) * d->n_nodes : nullptr,
                   n, visible);

  s.clear();
  vrows.clear();
  key_ids.clear();
  auto add_key = [&](const uint16_t* krow, const uint16_t* vrow, int id) {
    double dot = 0.0;
    for (int e = 0; e < D; ++e) dot += widen_bf16(qrow[e]) * widen_bf16(krow[e]);
    s.push_back(scale * dot);
    vrows.push_back(vrow);
    key_ids.push_back(id);
  };
  for (int j = 0; j < L; ++j)
    add_key(target_row(d, in.tk, in.page_table, c, kvh, j),
            in.tv ? target_row(d, in.tv, in.page_table, c, kvh, j) : nullptr, j);
  for (int m = 0; m < d->n_nodes; ++m)
    if (visible[m])
      add_key(draft_row(d, in.dk, c, kvh, m), in.dv ? draft_row(d, in.dv, c, kvh, m) : nullptr,
              L + m);
}

}  // namespace

extern "C" uint16_t kvo_round_bf16(double x) {
  // Direct round-to-nearest-even of x to 8 significant bits (no detour
  // through float, which could round twice).
  if (std::isnan(x)) return 0x7FC0;
  float f;
  uint32_t u;
  if (x == 0.0 || std::isinf(x)) {
    f = static_cast<float>(x);
    std::memcpy(&u, &f, 4);
    return static_cast<uint16_t>(u >> 16);
  }
  int e = std::ilogb(x);                 // |x| in [2^e, 2^(e+1))
  if (e < -126) e = -126;                // bf16 subnormal spacing is 2^-133
  double ulp = std::ldexp(1.0, e - 7);   // spacing of bf16 values in this binade
  const int old_mode = std::fegetround();
  std::fesetround(FE_TONEAREST);
  double r = std::nearbyint(x / ulp) * ulp;  // x / ulp is exact (power-of-two scale)
  std::fesetround(old_mode);
  const double bf16_max = 3.3895313892515355e38;  // (2 - 2^-7) * 2^127
  if (std::fabs(r) > bf16_max) r = std::copysign(INFINITY, x);
  f = static_cast<float>(r);            // exact: r has at most 8 significant bits
  std::memcpy(&u, &f, 4);
  return static_cast<uint16_t>(u >> 16);
}

extern "C" int kvo_attn(const kvo_desc* d, const uint16_t* q, const uint16_t* tk,
                        const uint16_t* tv, const int32_t* page_table, const int32_t* seq_lens,
                        const uint16_t* dk, const uint16_t* dv, const int32_t* tree_parent,
                        double* out, double* lse, int nthreads) {
  if (int rc = check_desc(d)) return rc;
  if (int rc = validate_contents(d, page_table, seq_lens, tree_parent)) return rc;
  const RowInputs in{d, q, tk, tv, dk, dv, page_table, seq_lens, tree_parent};
  const int D = d->head_dim;
  const long items = static_cast<long>(d->num_caches) * d->hq;
  std::atomic<long> next{0};

  auto worker = [&]() {
    std::vector<double> s;
    std::vector<const uint16_t*> vrows;
    std::vector<int> ids;
    std::vector<double> acc(D);
    for (long it = next.fetch_add(1); it < items; it = next.fetch_add(1)) {
      const int c = static_cast<int>(it / d->hq);
      const int h = static_cast<int>(it % d->hq);
      for (int nl = 0; nl < d->n_query; ++nl) {
        row_scores(in, c, nl, h, s, vrows, ids);
        double m = -INFINITY;
        for (double v : s) m = v > m ? v : m;
        double sum = 0.0;
        for (double v : s) sum += std::exp(v - m);
        const double row_lse = m + std::log(sum);
        std::fill(acc.begin(), acc.end(), 0.0);
        for (size_t j = 0; j < s.size(); ++j) {
          const double p = std::exp(s[j] - row_lse);
          for (int e = 0; e < D; ++e) acc[e] += p * widen_bf16(vrows[j][e]);
        }
        const size_t row = (static_cast<size_t>(c) * d->n_query + nl) * d->hq + h;
        for (int e = 0; e < D; ++e) out[row * D + e] = acc[e];
        lse[row] = row_lse;
      }
    }
  };

  int nt = nthreads > 0 ? nthreads : static_cast<int>(std::thread::hardware_concurrency());
  if (nt < 1) nt = 1;
  if (nt > items) nt = static_cast<int>(items > 0 ? items : 1);
  std::vector<std::thread> pool;
  for (int t = 1; t < nt; ++t) pool.emplace_back(worker);
  worker();
  for (auto& th : pool) th.join();
  return KVO_OK;
}

extern "C" int kvo_attn_probs(const kvo_desc* d, const uint16_t* q, const uint16_t* tk,
                              const int32_t* page_table, const int32_t* seq_lens,
                              const uint16_t* dk, const int32_t* tree_parent, int32_t c,
                              int32_t n_local, int32_t h, double* probs) {
  if (int rc = check_desc(d)) return rc;
  if (int rc = validate_contents(d, page_table, seq_lens, tree_parent)) return rc;
  if (c < 0 || c >= d->num_caches || n_local < 0 || n_local >= d->n_query || h < 0 || h >= d->hq)
    return KVO_ERR_SHAPE;
  const RowInputs in{d, q, tk, nullptr, dk, nullptr, page_table, seq_lens, tree_parent};
  std::vector<double> s;
  std::vector<const uint16_t*> vrows;
  std::vector<int> ids;
  row_scores(in, c, n_local, h, s, vrows, ids);
  double m = -INFINITY;
  for (double v : s) m = v > m ? v : m;
  double sum = 0.0;
  for (double v : s) sum += std::exp(v - m);
  const int total = seq_lens[c] + d->n_nodes;
  for (int j = 0; j < total; ++j) probs[j] = 0.0;
  for (size_t j = 0; j < s.size(); ++j) probs[ids[j]] = std::exp(s[j] - m) / sum;
  return KVO_OK;
}

extern "C" int kvo_append(const kvo_desc* d, const uint16_t* q_in, const uint16_t* k_in,
                          const uint16_t* v_in, const int32_t* positions, int32_t n0,
                          int32_t n_new, double rope_base, uint16_t* draft_k, uint16_t* draft_v,
                          uint16_t* q_out, double* q_rot_f64, double* k_rot_f64) {
  if (int rc = check_desc(d)) return rc;
  if (n0 < 0 || n_new < 0 || n0 + n_new > d->n_max || !(rope_base > 0.0)) return KVO_ERR_SHAPE;
  const int D = d->head_dim;
  const int half = D / 2;
  std::vector<double> x(D), y(D);

  auto rotate = [&](const uint16_t* src, int pos) {
    for (int e = 0; e < D; ++e) x[e] = widen_bf16(src[e]);
    for (int j = 0; j < half; ++j) {
      const double theta = pos * std::pow(rope_base, -2.0 * j / D);
      const double cs = std::cos(theta), sn = std::sin(theta);
      y[j] = x[j] * cs - x[j + half] * sn;
      y[j + half] = x[j + half] * cs + x[j] * sn;
    }
  };

  for (int c = 0; c < d->num_caches; ++c)
    for (int i = 0; i < n_new; ++i) {
      const int pos = positions[static_cast<size_t>(c) * n_new + i];
      for (int h = 0; h < d->hq; ++h) {
        const size_t off = ((static_cast<size_t>(c) * n_new + i) * d->hq + h) * D;
        rotate(q_in + off, pos);
        for (int e = 0; e < D; ++e) {
          q_out[off + e] = kvo_round_bf16(y[e]);
          if (q_rot_f64) q_rot_f64[off + e] = y[e];
        }
      }
      for (int h = 0; h < d->hkv; ++h) {
        const size_t off = ((static_cast<size_t>(c) * n_new + i) * d->hkv + h) * D;
        const size_t slot = ((static_cast<size_t>(c) * d->hkv + h) * d->n_max + n0 + i) * D;
        rotate(k_in + off, pos);
        for (int e = 0; e < D; ++e) {
          draft_k[slot + e] = kvo_round_bf16(y[e]);
          draft_v[slot + e] = v_in[off + e];
          if (k_rot_f64) k_rot_f64[off + e] = y[e];
        }
      }
    }
  return KVO_OK;
}
