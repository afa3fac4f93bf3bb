// Oracle for the embed-and-retrieve hot path of HeraSys' cross-workflow node
// merging.  TEST INFRASTRUCTURE ONLY: plain, slow, obviously correct CPU code
// that the GPU library is checked against.  Only the tests, the smoke check and
// the benchmark's CPU-baseline leg may load it; the product path never does.
// It shares no code, header, table or constant with the CUDA library.
//
// Each function follows a plain definition:
//   oracle_fnv1a64_bytes / oracle_fingerprint
//       the D_in part of the node signature Sig(v) (Section 3.3, Eq. 2), with
//       the hash H taken to be 64-bit FNV-1a over octets (the public FNV
//       specification: h <- (h xor octet) * prime mod 2^64, offset basis
//       14695981039346656037, prime 1099511628211).
//   oracle_unique_inverse
//       the merge step of topological fusion within a time window
//       (Section 3.3, "Dynamic Fusion and Reuse Mechanism" (I)) and the merge
//       sets M(v*) of Appendix A.2 ("Redundancy Elimination & Result
//       Sharing"): rows that are exactly equal form one node; the first
//       occurrence represents the group; every row keeps a pointer (inverse)
//       to its representative's ordinal.
//   oracle_topk
//       the vector-retrieval node of the RAG workloads (Section 4.1,
//       "Workloads": top-k chunks by similarity), as exact inner product in
//       fp64 over the bf16 inputs, ordered by descending score, ties to the
//       lower corpus index.
//   oracle_scatter
//       result sharing: the output of the kept node flows to every merged
//       node (Section 3.3 (I); Appendix A.2), dst[i] = src[map[i]].
//   oracle_segment_sum
//       the reuse-driven priority of a fused node (Section 3.3, "Reuse-Driven
//       Priority Adjustment", Eq. 3): phi(v*) is the sum of phi(v) over the
//       logical nodes v merged into v*, i.e. out[u] = sum of phi[i] over the
//       rows i with inverse[i] = u, added in fp64 in ascending row order.
//   oracle_rerank
//       the second stage of the RAG-with-rerank workflow (Section 4.1,
//       "Workloads": a reranker scores the initial top-12 chunks and the
//       top-8 by those scores are kept).  The reranker model is absent, so
//       its score is an exact fp64 inner product of bf16 rerank vectors; the
//       candidates of a query are ordered by descending score, ties to the
//       lower corpus index, and the first k2 kept.
//
// Parity pins for these functions live in tests/ (published FNV vectors,
// brute-force pairwise comparison, hand-computed top-k, library special
// cases, generator ground truth).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <numeric>
#include <thread>
#include <vector>

namespace {

// FNV-1a 64-bit parameters from the public FNV specification.
const uint64_t kOffsetBasis = 14695981039346656037ULL;
const uint64_t kPrime = 1099511628211ULL;

// Length of row i, or -1 if the length is outside [0, stride].
int64_t row_len(const int32_t* lens, int64_t i, int32_t stride) {
  int64_t len = lens ? (int64_t)lens[i] : (int64_t)stride;
  if (len < 0 || len > stride) return -1;
  return len;
}

// bf16 bit pattern -> double, exactly: a bf16 value is the upper half of an
// IEEE binary32 value.
double bf16_to_double(uint16_t bits) {
  uint32_t w = (uint32_t)bits << 16;
  float f;
  std::memcpy(&f, &w, sizeof f);
  return (double)f;
}

}  // namespace

extern "C" {

uint64_t oracle_fnv_offset_basis(void) { return kOffsetBasis; }

// FNV-1a over nbytes octets, starting from the state h0 (pass the offset
// basis for the standard hash; pass an earlier result to continue a hash
// over a concatenation).
uint64_t oracle_fnv1a64_bytes(const uint8_t* p, int64_t nbytes, uint64_t h0) {
  uint64_t h = h0;
  for (int64_t i = 0; i < nbytes; ++i) {
    h ^= (uint64_t)p[i];
    h *= kPrime;  // unsigned arithmetic: mod 2^64
  }
  return h;
}

// fp[i] = FNV-1a(seed, little-endian octets of tokens[i, 0:len_i]).
// tokens is row-major [n, stride]; lens == NULL means every row has length
// stride.  Returns 0, or 1 if some length is outside [0, stride].
int oracle_fingerprint(const int32_t* tokens, int64_t n, int32_t stride,
                       const int32_t* lens, uint64_t seed, uint64_t* fp_out) {
  for (int64_t i = 0; i < n; ++i) {
    int64_t len = row_len(lens, i, stride);
    if (len < 0) return 1;
    std::vector<uint8_t> octets((size_t)len * 4);
    for (int64_t t = 0; t < len; ++t) {
      uint32_t w = (uint32_t)tokens[i * (int64_t)stride + t];
      // Little-endian: least significant octet first, independent of the
      // host's byte order.
      octets[4 * t + 0] = (uint8_t)(w & 0xffu);
      octets[4 * t + 1] = (uint8_t)((w >> 8) & 0xffu);
      octets[4 * t + 2] = (uint8_t)((w >> 16) & 0xffu);
      octets[4 * t + 3] = (uint8_t)((w >> 24) & 0xffu);
    }
    fp_out[i] = oracle_fnv1a64_bytes(octets.data(), (int64_t)octets.size(), seed);
  }
  return 0;
}

// Exact unique with inverse.  Two rows are equal iff they have the same length
// and the same tokens in [0, len); tokens beyond len are ignored.  Groups are
// represented by their first occurrence; unique_idx lists the representatives
// in ascending index order; inverse[i] is the ordinal of row i's group in that
// list.  The fingerprints play no part in the definition: the result depends
// on row content alone.  Returns 0, or 1 if some length is out of range.
int oracle_unique_inverse(const int32_t* tokens, int64_t n, int32_t stride,
                          const int32_t* lens, int32_t* n_unique_out,
                          int32_t* unique_idx_out, int32_t* inverse_out) {
  std::vector<int64_t> len(n);
  for (int64_t i = 0; i < n; ++i) {
    len[i] = row_len(lens, i, stride);
    if (len[i] < 0) return 1;
  }
  // Order rows by (length, tokens lexicographically, index): equal rows
  // become adjacent and each run starts with its smallest index.
  auto row = [&](int64_t i) { return tokens + i * (int64_t)stride; };
  std::vector<int64_t> order(n);
  std::iota(order.begin(), order.end(), 0);
  std::sort(order.begin(), order.end(), [&](int64_t a, int64_t b) {
    if (len[a] != len[b]) return len[a] < len[b];
    const int32_t* ra = row(a);
    const int32_t* rb = row(b);
    for (int64_t t = 0; t < len[a]; ++t)
      if (ra[t] != rb[t]) return ra[t] < rb[t];
    return a < b;
  });
  auto same = [&](int64_t a, int64_t b) {
    if (len[a] != len[b]) return false;
    return std::equal(row(a), row(a) + len[a], row(b));
  };
  std::vector<int64_t> rep(n);
  for (int64_t p = 0; p < n; ++p) {
    int64_t i = order[p];
    if (p > 0 && same(order[p - 1], i))
      rep[i] = rep[order[p - 1]];
    else
      rep[i] = i;  // first of its run: the smallest index of the group
  }
  // Ordinals in first-occurrence order.
  std::vector<int32_t> ordinal(n, -1);
  int32_t next = 0;
  for (int64_t i = 0; i < n; ++i) {
    if (rep[i] == i) {
      ordinal[i] = next;
      unique_idx_out[next] = (int32_t)i;
      ++next;
    }
  }
  for (int64_t i = 0; i < n; ++i) inverse_out[i] = ordinal[rep[i]];
  *n_unique_out = next;
  return 0;
}

// Exact top-k by inner product.  queries [nq, d] and corpus [N, d] are bf16
// bit patterns, row-major.  For each query q: s[j] = sum_t Q[q,t] * C[j,t]
// summed in fp64 in order t = 0..d-1; the result lists the k pairs (s, j)
// that come first in the order (s descending, j ascending).  Queries are
// spread over nthreads host threads (0: all hardware threads).  Returns 0, or
// 1 if k is outside [1, N].
int oracle_topk(const uint16_t* queries, int64_t nq, const uint16_t* corpus,
                int64_t N, int32_t d, int32_t k, double* scores_out,
                int32_t* ids_out, int32_t nthreads) {
  if (k < 1 || (int64_t)k > N) return 1;
  if (nthreads <= 0) nthreads = (int32_t)std::max(1u, std::thread::hardware_concurrency());
  if ((int64_t)nthreads > nq) nthreads = (int32_t)std::max<int64_t>(1, nq);
  auto one_query = [&](int64_t q) {
    std::vector<double> qv(d);
    for (int32_t t = 0; t < d; ++t) qv[t] = bf16_to_double(queries[q * d + t]);
    std::vector<double> s(N);
    for (int64_t j = 0; j < N; ++j) {
      const uint16_t* c = corpus + j * (int64_t)d;
      double acc = 0.0;
      for (int32_t t = 0; t < d; ++t) acc += qv[t] * bf16_to_double(c[t]);
      s[j] = acc;
    }
    std::vector<int64_t> idx(N);
    std::iota(idx.begin(), idx.end(), 0);
    std::partial_sort(idx.begin(), idx.begin() + k, idx.end(),
                      [&](int64_t a, int64_t b) {
                        if (s[a] != s[b]) return s[a] > s[b];
                        return a < b;
                      });
    for (int32_t r = 0; r < k; ++r) {
      scores_out[q * k + r] = s[idx[r]];
      ids_out[q * k + r] = (int32_t)idx[r];
    }
  };
  std::vector<std::thread> pool;
  for (int32_t w = 0; w < nthreads; ++w)
    pool.emplace_back([&, w] {
      for (int64_t q = w; q < nq; q += nthreads) one_query(q);
    });
  for (auto& th : pool) th.join();
  return 0;
}

// Exact fp64 inner products for an explicit list of (query, corpus row)
// pairs: out[p] = sum_t Q[qi[p], t] * C[cj[p], t], in order t = 0..d-1.  Used
// to score the ids a GPU run returned.
void oracle_pair_scores(const uint16_t* queries, const uint16_t* corpus,
                        int32_t d, const int64_t* qi, const int64_t* cj,
                        int64_t npairs, double* out) {
  for (int64_t p = 0; p < npairs; ++p) {
    const uint16_t* a = queries + qi[p] * (int64_t)d;
    const uint16_t* b = corpus + cj[p] * (int64_t)d;
    double acc = 0.0;
    for (int32_t t = 0; t < d; ++t) acc += bf16_to_double(a[t]) * bf16_to_double(b[t]);
    out[p] = acc;
  }
}

// dst[i, :] = src[map[i], :] for rows of row_bytes bytes.  Returns 0, or 1 if
// some map entry is outside [0, n_src).
int oracle_scatter(const uint8_t* src, int64_t n_src, int64_t row_bytes,
                   const int32_t* map, int64_t n, uint8_t* dst) {
  for (int64_t i = 0; i < n; ++i) {
    if (map[i] < 0 || (int64_t)map[i] >= n_src) return 1;
    std::memcpy(dst + i * row_bytes, src + (int64_t)map[i] * row_bytes, (size_t)row_bytes);
  }
  return 0;
}

// For each query q: the candidates cand[q, 0:k1] (entries < 0 are absent)
// scored by the fp64 inner product of rq[q] and rc[id], ordered by (score
// descending, id ascending), the first k2 written to scores_out / ids_out
// (-inf / -1 past the number of present candidates).  Returns 0, or 1 if a
// candidate id is >= n_rc.
int oracle_rerank(const uint16_t* rq, int64_t nq, const uint16_t* rc, int64_t n_rc, int32_t d,
                  const int32_t* cand, int32_t k1, int32_t k2, double* scores_out,
                  int32_t* ids_out) {
  for (int64_t q = 0; q < nq; ++q) {
    std::vector<std::pair<double, int32_t>> c;
    for (int32_t j = 0; j < k1; ++j) {
      const int32_t id = cand[q * k1 + j];
      if (id < 0) continue;
      if ((int64_t)id >= n_rc) return 1;
      double s = 0.0;
      for (int32_t t = 0; t < d; ++t)
        s += bf16_to_double(rq[q * d + t]) * bf16_to_double(rc[(int64_t)id * d + t]);
      c.push_back({s, id});
    }
    std::sort(c.begin(), c.end(), [](const std::pair<double, int32_t>& a,
                                     const std::pair<double, int32_t>& b) {
      return a.first != b.first ? a.first > b.first : a.second < b.second;
    });
    for (int32_t j = 0; j < k2; ++j) {
      const bool have = j < (int32_t)c.size();
      scores_out[q * k2 + j] = have ? c[j].first : -INFINITY;
      ids_out[q * k2 + j] = have ? c[j].second : -1;
    }
  }
  return 0;
}

// out[u] = sum over rows i with inverse[i] == u of phi[i], for u in
// [0, n_groups); a group without rows sums to 0.  Returns 0, or 1 if some
// inverse entry is outside [0, n_groups).
int oracle_segment_sum(const double* phi, const int32_t* inverse, int64_t n, int64_t n_groups,
                       double* out) {
  for (int64_t u = 0; u < n_groups; ++u) out[u] = 0.0;
  for (int64_t i = 0; i < n; ++i) {
    if (inverse[i] < 0 || (int64_t)inverse[i] >= n_groups) return 1;
    out[inverse[i]] += phi[i];
  }
  return 0;
}

}  // extern "C"
