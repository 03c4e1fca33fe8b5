// The prompt pre-scorer (Pro-Router, Section 3.1, Eq. 2) on the host CPU, as
// the paper keeps it off the accelerator:
//
//   p_pre(x) = sigmoid(w . phi(x) + b),  phi(x) = [TF-IDF(prompt), image count, length]
//
// pr_prescorer_fit builds the vocabulary and the smoothed idf of a corpus;
// pr_prescorer_score scores a batch of prompts, in parallel over host
// threads.  Readings of what the paper leaves open (the same as the float64
// reference used by the tests):
//   * a token is a maximal run of word bytes ([0-9A-Za-z_] and every byte >=
//     0x80) at least two bytes long, ASCII letters lowercased;
//   * the vocabulary holds every corpus term with document frequency >=
//     min_df, columns in byte order of the terms;
//   * tf = raw count, idf = ln((1 + n) / (1 + df)) + 1, the row scaled to unit
//     Euclidean length (a row without vocabulary terms stays zero);
//   * length = the prompt's token count; w = V TF-IDF weights, then the
//     image-count weight, then the length weight.
// Sums run in double precision in ascending column order.
//
// Both fitting and scoring hash each token while it is read (64-bit FNV-1a
// over the lowercased bytes).  Fitting counts document frequencies in an
// open-addressing table of the corpus's terms; scoring finds a token's column
// in an open-addressing table of the vocabulary and counts it in a per-thread
// dense array, so that no token is copied into a string or a node-based map.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <memory>
#include <new>
#include <string>
#include <thread>
#include <utility>
#include <vector>

#include "pro_router.h"

struct pr_prescorer {
  std::vector<std::string> terms;  // column -> term, byte order
  std::vector<double> idf;
  int64_t n_docs = 0;
  // term -> column: open addressing, linear probing, at most half full
  std::vector<uint64_t> slot_hash;
  std::vector<int32_t> slot_col;  // -1: empty
  uint64_t slot_mask = 0;
};

namespace {

inline bool word_byte(unsigned char c) {
  return (c >= '0' && c <= '9') || (c >= 'a' && c <= 'z') || (c >= 'A' && c <= 'Z') || c == '_' ||
         c >= 0x80;
}

constexpr uint64_t FNV_OFFSET = 1469598103934665603ull, FNV_PRIME = 1099511628211ull;

inline uint64_t fnv1a(const char* p, size_t n) {
  uint64_t h = FNV_OFFSET;
  for (size_t i = 0; i < n; ++i) h = (h ^ (unsigned char)p[i]) * FNV_PRIME;
  return h;
}

inline unsigned char lower(unsigned char c) {
  return (c >= 'A' && c <= 'Z') ? (unsigned char)(c + ('a' - 'A')) : c;
}

// per byte: 0 outside a token (the NUL included), else the byte lowercased
struct ByteClass {
  unsigned char v[256];
  ByteClass() {
    for (int c = 0; c < 256; ++c) v[c] = (c != 0 && word_byte((unsigned char)c)) ? lower((unsigned char)c) : 0;
  }
};
const ByteClass kByte;

// calls f(tok, n, h) for every token of the NUL-terminated text: tok[0, n)
// its lowercased bytes (in buf, reused), h their FNV-1a hash, both formed
// as the bytes are read
template <class F>
void scan_tokens(const char* text, std::vector<unsigned char>& buf, F&& f) {
  size_t n = 0;
  uint64_t h = FNV_OFFSET;
  for (const unsigned char* p = reinterpret_cast<const unsigned char*>(text);; ++p) {
    const unsigned char c = *p;
    const unsigned char lc = kByte.v[c];
    if (lc != 0) {
      if (n == buf.size()) buf.resize(buf.empty() ? 64 : 2 * buf.size());
      buf[n++] = lc;
      h = (h ^ lc) * FNV_PRIME;
      continue;
    }
    if (n >= 2) f(static_cast<const unsigned char*>(buf.data()), n, h);
    n = 0;
    h = FNV_OFFSET;
    if (c == 0) break;
  }
}

// The corpus's distinct terms while fitting: open addressing over the terms'
// hashes, each term's document frequency and the last document that counted
// it (a document counts a term once).
struct TermCounter {
  std::vector<std::string> terms;
  std::vector<int64_t> df;
  std::vector<int32_t> last_doc;
  std::vector<uint64_t> slot_hash;
  std::vector<int32_t> slot_id;  // -1: empty
  uint64_t mask = 0;

  TermCounter() { rehash(1024); }
  void rehash(size_t cap) {
    slot_hash.assign(cap, 0ull);
    slot_id.assign(cap, -1);
    mask = cap - 1;
    for (size_t j = 0; j < terms.size(); ++j) {
      const uint64_t h = fnv1a(terms[j].data(), terms[j].size());
      uint64_t i = h & mask;
      while (slot_id[i] >= 0) i = (i + 1) & mask;
      slot_hash[i] = h;
      slot_id[i] = (int32_t)j;
    }
  }
  void count(const unsigned char* tok, size_t n, uint64_t h, int32_t doc) {
    uint64_t i = h & mask;
    for (;; i = (i + 1) & mask) {
      const int32_t id = slot_id[i];
      if (id < 0) break;
      const std::string& t = terms[(size_t)id];
      if (slot_hash[i] == h && t.size() == n && std::memcmp(t.data(), tok, n) == 0) {
        if (last_doc[(size_t)id] != doc) {
          last_doc[(size_t)id] = doc;
          ++df[(size_t)id];
        }
        return;
      }
    }
    terms.emplace_back(reinterpret_cast<const char*>(tok), n);
    df.push_back(1);
    last_doc.push_back(doc);
    slot_hash[i] = h;
    slot_id[i] = (int32_t)(terms.size() - 1);
    if (2 * terms.size() > slot_id.size()) rehash(2 * slot_id.size());
  }
};

// the column of the lowercased token tok[0, n) with hash h, or -1
inline int32_t find_column(const pr_prescorer& ps, const unsigned char* tok, size_t n, uint64_t h) {
  if (ps.slot_col.empty()) return -1;
  for (uint64_t i = h & ps.slot_mask;; i = (i + 1) & ps.slot_mask) {
    const int32_t c = ps.slot_col[i];
    if (c < 0) return -1;
    if (ps.slot_hash[i] == h) {
      const std::string& t = ps.terms[(size_t)c];
      if (t.size() == n && std::memcmp(t.data(), tok, n) == 0) return c;
    }
  }
}

void build_table(pr_prescorer& ps) {
  size_t cap = 16;
  while (cap < 2 * ps.terms.size()) cap <<= 1;
  ps.slot_hash.assign(cap, 0ull);
  ps.slot_col.assign(cap, -1);
  ps.slot_mask = cap - 1;
  for (size_t j = 0; j < ps.terms.size(); ++j) {
    const uint64_t h = fnv1a(ps.terms[j].data(), ps.terms[j].size());
    uint64_t i = h & ps.slot_mask;
    while (ps.slot_col[i] >= 0) i = (i + 1) & ps.slot_mask;
    ps.slot_hash[i] = h;
    ps.slot_col[i] = (int32_t)j;
  }
}

struct Row {
  std::vector<std::pair<int32_t, double>> v;  // (column, value), ascending column
  int64_t length = 0;
  std::vector<int32_t> count;    // per column (all zero between prompts)
  std::vector<int32_t> touched;  // columns counted in this prompt
  std::vector<unsigned char> tok;
};

void tfidf_row(const pr_prescorer& ps, const char* prompt, Row& row) {
  if (row.count.size() != ps.terms.size()) row.count.assign(ps.terms.size(), 0);
  row.touched.clear();
  row.length = 0;
  scan_tokens(prompt, row.tok, [&](const unsigned char* tok, size_t n, uint64_t h) {
    ++row.length;
    const int32_t col = find_column(ps, tok, n, h);
    if (col >= 0 && row.count[(size_t)col]++ == 0) row.touched.push_back(col);
  });
  std::sort(row.touched.begin(), row.touched.end());
  row.v.clear();
  row.v.reserve(row.touched.size());
  for (const int32_t col : row.touched) {
    row.v.emplace_back(col, (double)row.count[(size_t)col] * ps.idf[(size_t)col]);
    row.count[(size_t)col] = 0;
  }
  double ss = 0.0;
  for (const auto& e : row.v) ss += e.second * e.second;
  if (ss > 0.0) {
    const double inv = 1.0 / std::sqrt(ss);
    for (auto& e : row.v) e.second *= inv;
  }
}

double row_logit(const pr_prescorer& ps, const Row& row, int32_t n_images, const float* w,
                 float b) {
  const size_t V = ps.terms.size();
  double z = (double)b;
  for (const auto& e : row.v) z += (double)w[e.first] * e.second;
  z += (double)w[V] * (double)n_images + (double)w[V + 1] * (double)row.length;
  return z;
}

double sigmoid(double z) {
  if (z >= 0.0) return 1.0 / (1.0 + std::exp(-z));
  const double e = std::exp(z);
  return e / (1.0 + e);
}

}  // namespace

extern "C" {

pr_status pr_prescorer_fit(const char* const* docs, int32_t n_docs, int32_t min_df,
                           pr_prescorer** out) {
  if (!out) return PR_ERR_INVALID_ARG;
  *out = nullptr;
  if (n_docs < 0 || (n_docs > 0 && !docs) || min_df < 1) return PR_ERR_INVALID_ARG;
  for (int32_t i = 0; i < n_docs; ++i)
    if (!docs[i]) return PR_ERR_INVALID_ARG;
  try {
    TermCounter tc;
    std::vector<unsigned char> buf;
    for (int32_t i = 0; i < n_docs; ++i)
      scan_tokens(docs[i], buf,
                  [&](const unsigned char* tok, size_t n, uint64_t h) { tc.count(tok, n, h, i); });
    // the terms kept, in byte order (std::string compares as unsigned char)
    std::vector<int32_t> keep;
    for (size_t j = 0; j < tc.terms.size(); ++j)
      if (tc.df[j] >= min_df) keep.push_back((int32_t)j);
    std::sort(keep.begin(), keep.end(),
              [&](int32_t x, int32_t y) { return tc.terms[(size_t)x] < tc.terms[(size_t)y]; });
    std::unique_ptr<pr_prescorer> ps(new pr_prescorer);
    ps->terms.reserve(keep.size());
    ps->idf.reserve(keep.size());
    for (const int32_t j : keep) {
      ps->terms.push_back(std::move(tc.terms[(size_t)j]));
      ps->idf.push_back(std::log((1.0 + (double)n_docs) / (1.0 + (double)tc.df[(size_t)j])) + 1.0);
    }
    ps->n_docs = n_docs;
    build_table(*ps);
    *out = ps.release();
    return PR_OK;
  } catch (const std::bad_alloc&) {
    return PR_ERR_NO_MEMORY;
  }
}

void pr_prescorer_destroy(pr_prescorer* ps) { delete ps; }

int64_t pr_prescorer_vocab_size(const pr_prescorer* ps) {
  return ps ? (int64_t)ps->terms.size() : -1;
}

const char* pr_prescorer_term(const pr_prescorer* ps, int64_t column) {
  if (!ps || column < 0 || column >= (int64_t)ps->terms.size()) return nullptr;
  return ps->terms[(size_t)column].c_str();
}

pr_status pr_prescorer_features(const pr_prescorer* ps, const char* prompt, int32_t cap,
                                int32_t* columns, float* values, int32_t* nnz, int64_t* length) {
  if (!ps || !prompt || cap < 0 || !nnz || !length || (cap > 0 && (!columns || !values)))
    return PR_ERR_INVALID_ARG;
  try {
    Row row;
    tfidf_row(*ps, prompt, row);
    *nnz = (int32_t)row.v.size();
    *length = row.length;
    if ((int64_t)row.v.size() > cap) return PR_ERR_INVALID_ARG;
    for (size_t i = 0; i < row.v.size(); ++i) {
      columns[i] = row.v[i].first;
      values[i] = (float)row.v[i].second;
    }
    return PR_OK;
  } catch (const std::bad_alloc&) {
    return PR_ERR_NO_MEMORY;
  }
}

pr_status pr_prescorer_score(const pr_prescorer* ps, const char* const* prompts,
                             const int32_t* n_images, int32_t n, const float* w, float b,
                             int32_t n_threads, float* score, float* logit) {
  if (!ps || n < 0 || !w || n_threads < 0) return PR_ERR_INVALID_ARG;
  if (n == 0) return PR_OK;
  if (!prompts || !n_images || !score) return PR_ERR_INVALID_ARG;
  for (int32_t i = 0; i < n; ++i)
    if (!prompts[i] || n_images[i] < 0) return PR_ERR_INVALID_ARG;
  int nt = n_threads > 0 ? n_threads : (int)std::max(1u, std::thread::hardware_concurrency());
  nt = std::max(1, std::min(nt, n));
  bool failed = false;
  auto work = [&](int32_t lo, int32_t hi, bool* fail) {
    try {
      Row row;
      for (int32_t i = lo; i < hi; ++i) {
        tfidf_row(*ps, prompts[i], row);
        const double z = row_logit(*ps, row, n_images[i], w, b);
        score[i] = (float)sigmoid(z);
        if (logit) logit[i] = (float)z;
      }
    } catch (const std::bad_alloc&) {
      *fail = true;
    }
  };
  if (nt == 1) {
    work(0, n, &failed);
    return failed ? PR_ERR_NO_MEMORY : PR_OK;
  }
  std::vector<std::thread> th;
  std::vector<char> fails((size_t)nt, 0);
  try {
    th.reserve((size_t)nt);
    for (int t = 0; t < nt; ++t) {
      const int32_t lo = (int32_t)((int64_t)n * t / nt), hi = (int32_t)((int64_t)n * (t + 1) / nt);
      th.emplace_back([&, lo, hi, t] {
        bool f = false;
        work(lo, hi, &f);
        fails[(size_t)t] = f;
      });
    }
  } catch (...) {
    for (auto& x : th) x.join();
    return PR_ERR_NO_MEMORY;
  }
  for (auto& x : th) x.join();
  for (char f : fails)
    if (f) return PR_ERR_NO_MEMORY;
  return PR_OK;
}

}  // extern "C"
