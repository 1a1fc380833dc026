// Archer denoising-step oracle: plain, slow, fp64 CPU statement of what the
// hot path computes.
//
// TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the bench's
// CPU-baseline leg load this library.  It shares no code, header, table or
// helper with the CUDA path, and the CUDA path never calls it.
//
// Every floating-point result is computed in IEEE double from inputs that the
// caller widened exactly (bf16 -> fp64, fp32 -> fp64).  Nothing is blocked,
// fused or reordered beyond the plain definitions cited at each function.
//
// Pins (what fixes each function independently of this file) live in
// tests/test_oracle_pins.py: closed forms, mpmath brute force, exhaustive
// enumeration and the paper's refresh-every-step == eager identity.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <thread>
#include <vector>

namespace {

// Run body(i) for i in [0, n) on up to n_threads std::threads.
template <class F>
void parallel_for(int64_t n, int n_threads, F body) {
  if (n_threads <= 0) n_threads = (int)std::max(1u, std::thread::hardware_concurrency());
  if (n_threads > n) n_threads = (int)std::max<int64_t>(1, n);
  if (n_threads == 1) {
    for (int64_t i = 0; i < n; ++i) body(i);
    return;
  }
  std::vector<std::thread> pool;
  pool.reserve(n_threads);
  for (int t = 0; t < n_threads; ++t) {
    pool.emplace_back([=, &body]() {
      for (int64_t i = t; i < n; i += n_threads) body(i);
    });
  }
  for (auto& th : pool) th.join();
}

// One query row of Attn(q, K_cat, V_cat) with the explicit concatenation
// K_cat = [K_p || K_g], V_cat = [V_p || V_g] already built (Sec. 4.1,
// Eq. archer-attention): non-causal, every key visible.
//   s_j   = scale * <q, k_j>
//   m     = max_j s_j
//   p_j   = exp(s_j - m) / sum_k exp(s_k - m)
//   out   = sum_j p_j v_j
//   lse   = m + log sum_k exp(s_k - m)
void attend_row(const double* q, const std::vector<double>& kcat,
                const std::vector<double>& vcat, int n_keys, int d, double scale,
                double* out, double* lse, double* probs_out) {
  std::vector<double> s(n_keys);
  for (int j = 0; j < n_keys; ++j) {
    double dot = 0.0;
    for (int c = 0; c < d; ++c) dot += q[c] * kcat[(size_t)j * d + c];
    s[j] = scale * dot;
  }
  double m = -std::numeric_limits<double>::infinity();
  for (int j = 0; j < n_keys; ++j) m = std::max(m, s[j]);
  std::vector<double> e(n_keys);
  double sum = 0.0;
  for (int j = 0; j < n_keys; ++j) {
    e[j] = std::exp(s[j] - m);
    sum += e[j];
  }
  std::vector<double> p(n_keys);
  for (int j = 0; j < n_keys; ++j) p[j] = e[j] / sum;
  for (int c = 0; c < d; ++c) out[c] = 0.0;
  for (int j = 0; j < n_keys; ++j)
    for (int c = 0; c < d; ++c) out[c] += p[j] * vcat[(size_t)j * d + c];
  if (lse) *lse = m + std::log(sum);
  if (probs_out)
    for (int j = 0; j < n_keys; ++j) probs_out[j] = p[j];
}

// Build [K_p || K_g] (and the same for V) for sequence b, KV head kvh.
void concat_kv(int b, int kvh, int P, int G, int Hkv, int D, const double* kp,
               const double* vp, const double* kg, const double* vg,
               std::vector<double>& kcat, std::vector<double>& vcat) {
  const int N = P + G;
  kcat.assign((size_t)N * D, 0.0);
  vcat.assign((size_t)N * D, 0.0);
  for (int j = 0; j < P; ++j) {
    const size_t src = (((size_t)b * P + j) * Hkv + kvh) * D;
    std::memcpy(&kcat[(size_t)j * D], kp + src, sizeof(double) * D);
    std::memcpy(&vcat[(size_t)j * D], vp + src, sizeof(double) * D);
  }
  for (int j = 0; j < G; ++j) {
    const size_t src = (((size_t)b * G + j) * Hkv + kvh) * D;
    std::memcpy(&kcat[(size_t)(P + j) * D], kg + src, sizeof(double) * D);
    std::memcpy(&vcat[(size_t)(P + j) * D], vg + src, sizeof(double) * D);
  }
}

}  // namespace

extern "C" {

// Attention of M query rows over the explicit concatenation of a prompt
// segment (P rows) and a response segment (G rows), per (sequence, head).
// GQA: query head h reads KV head h / (Hq / Hkv).
//   q   [B, M, Hq, D]      kp, vp [B, P, Hkv, D]     kg, vg [B, G, Hkv, D]
//   out [B, M, Hq, D]      lse [B, Hq, M] (may be null)
// Only rows with row_begin[b] <= i < M are computed (row_begin may be null:
// all rows); other rows of out / lse are left untouched.
// Returns 0, or -1 on a bad argument.
int oracle_attention(int B, int M, int P, int G, int Hq, int Hkv, int D, double scale,
                     const double* q, const double* kp, const double* vp,
                     const double* kg, const double* vg, const int32_t* row_begin,
                     double* out, double* lse, int n_threads) {
  if (B < 0 || M < 0 || P < 0 || G < 0 || Hq <= 0 || Hkv <= 0 || D <= 0) return -1;
  if (Hq % Hkv != 0 || P + G <= 0) return -1;
  const int group = Hq / Hkv;
  const int N = P + G;
  parallel_for((int64_t)B * Hq, n_threads, [&](int64_t bh) {
    const int b = (int)(bh / Hq), h = (int)(bh % Hq);
    const int kvh = h / group;
    std::vector<double> kcat, vcat;
    concat_kv(b, kvh, P, G, Hkv, D, kp, vp, kg, vg, kcat, vcat);
    const int i0 = row_begin ? row_begin[b] : 0;
    for (int i = std::max(0, i0); i < M; ++i) {
      const size_t qo = (((size_t)b * M + i) * Hq + h) * D;
      double l = 0.0;
      attend_row(q + qo, kcat, vcat, N, D, scale, out + qo, &l, nullptr);
      if (lse) lse[((size_t)b * Hq + h) * M + i] = l;
    }
  });
  return 0;
}

// Cached response step (Sec. 4.1, Eq. archer-cached / archer-attention):
// the G response queries attend over [K_p(g_r) || K_g(g_t)], i.e. the cached
// prompt K/V of the anchor and the fresh response K/V.
//   q_resp [B, G, Hq, D]; k_cache, v_cache [B, P, Hkv, D]; k_resp, v_resp [B, G, Hkv, D]
//   out [B, G, Hq, D]; lse [B, Hq, G] (nullable)
int oracle_attn_step(int B, int P, int G, int Hq, int Hkv, int D, double scale,
                     const double* q_resp, const double* k_cache, const double* v_cache,
                     const double* k_resp, const double* v_resp, double* out, double* lse,
                     int n_threads) {
  return oracle_attention(B, G, P, G, Hq, Hkv, D, scale, q_resp, k_cache, v_cache, k_resp,
                          v_resp, nullptr, out, lse, n_threads);
}

// Prompt refresh (Sec. 4.2; Algorithm 1's FullForward): for every sequence
// whose flag is set (all sequences when flags is null), all N = P + G
// positions are queries over the fresh [K_p(g_t) || K_g(g_t)], and the prompt
// cache is replaced by the fresh prompt K/V (C_r <- C_p(g_t)).  A sequence
// whose flag is clear takes the cached step instead: its response queries
// (rows P..N-1 of q_all) attend over [K_cache || K_g]; its prompt rows of out
// and lse are left untouched and its cache is kept.
//   q_all [B, N, Hq, D]; k_new, v_new [B, P, Hkv, D]; k_resp, v_resp [B, G, Hkv, D]
//   k_cache, v_cache [B, P, Hkv, D] (read for clear flags, written for set flags)
//   out [B, N, Hq, D]; lse [B, Hq, N] (nullable)
int oracle_prompt_refresh(int B, int P, int G, int Hq, int Hkv, int D, double scale,
                          const double* q_all, const double* k_new, const double* v_new,
                          const double* k_resp, const double* v_resp, double* out,
                          double* lse, double* k_cache, double* v_cache,
                          const uint8_t* flags, int n_threads) {
  if (B < 0 || P < 0 || G <= 0) return -1;
  const int N = P + G;
  const size_t per_seq = (size_t)P * Hkv * D;
  for (int b = 0; b < B; ++b) {
    const bool refresh = flags == nullptr || flags[b] != 0;
    // One sequence at a time keeps each call a plain instance of the definition.
    const double* kp = refresh ? k_new + b * per_seq : k_cache + b * per_seq;
    const double* vp = refresh ? v_new + b * per_seq : v_cache + b * per_seq;
    const size_t q_off = (size_t)b * N * Hq * D;
    const size_t g_off = (size_t)b * G * Hkv * D;
    std::vector<double> lse_b(lse ? (size_t)Hq * N : 0);
    const int32_t begin = refresh ? 0 : P;
    if (lse)
      for (int h = 0; h < Hq; ++h)
        for (int i = 0; i < N; ++i) lse_b[(size_t)h * N + i] = lse[((size_t)b * Hq + h) * N + i];
    int rc = oracle_attention(1, N, P, G, Hq, Hkv, D, scale, q_all + q_off, kp, vp,
                              k_resp + g_off, v_resp + g_off, &begin, out + q_off,
                              lse ? lse_b.data() : nullptr, n_threads);
    if (rc != 0) return rc;
    if (lse)
      for (int h = 0; h < Hq; ++h)
        for (int i = 0; i < N; ++i) lse[((size_t)b * Hq + h) * N + i] = lse_b[(size_t)h * N + i];
    if (refresh && k_cache != k_new) {
      std::memcpy(k_cache + b * per_seq, k_new + b * per_seq, sizeof(double) * per_seq);
      std::memcpy(v_cache + b * per_seq, v_new + b * per_seq, sizeof(double) * per_seq);
    }
  }
  return 0;
}

// The explicit softmax row p_j (j over [prompt || response] keys) of one query
// (b, h, i) of oracle_attention; used to check that rows sum to one.
int oracle_attention_probs(int P, int G, int Hq, int Hkv, int D, double scale,
                           const double* q_row, const double* kp, const double* vp,
                           const double* kg, const double* vg, int h, double* probs) {
  if (Hq % Hkv != 0 || h < 0 || h >= Hq) return -1;
  const int kvh = h / (Hq / Hkv);
  std::vector<double> kcat, vcat, out(D);
  concat_kv(0, kvh, P, G, Hkv, D, kp, vp, kg, vg, kcat, vcat);
  attend_row(q_row, kcat, vcat, P + G, D, scale, out.data(), nullptr, probs);
  return 0;
}

// Decoder scoring of one row of logits (the inputs the rollback decoder's
// confidence rule reads; Sec. 6 "confidence", Eq. theory-margin):
//   p = softmax(z)  (explicit vector)
//   top1 = the lowest index attaining max_j z_j
//   top2 = the index after top1 in (value desc, index asc) order
//   max_prob = p[top1]; margin = p[top1] - p[top2]  (p[top2] := 0 when V == 1)
//   cur_prob = p[cur] for an unmasked position with a valid current token, else 0
int oracle_decode_scores(int rows, int V, const double* z, int64_t row_stride,
                         const uint8_t* mask_state, const int32_t* cur_tokens,
                         double* max_prob, int32_t* top1, double* margin, int32_t* top2,
                         double* cur_prob, int n_threads) {
  if (rows < 0 || V <= 0 || row_stride < V) return -1;
  parallel_for(rows, n_threads, [&](int64_t r) {
    const double* zr = z + r * row_stride;
    double m = -std::numeric_limits<double>::infinity();
    for (int j = 0; j < V; ++j) m = std::max(m, zr[j]);
    std::vector<double> p(V);
    double sum = 0.0;
    for (int j = 0; j < V; ++j) {
      p[j] = std::exp(zr[j] - m);
      sum += p[j];
    }
    for (int j = 0; j < V; ++j) p[j] /= sum;
    int t1 = -1;
    for (int j = 0; j < V; ++j)
      if (t1 < 0 || zr[j] > zr[t1]) t1 = j;
    int t2 = -1;
    for (int j = 0; j < V; ++j) {
      if (j == t1) continue;
      if (t2 < 0 || zr[j] > zr[t2]) t2 = j;
    }
    max_prob[r] = p[t1];
    top1[r] = t1;
    margin[r] = p[t1] - (t2 >= 0 ? p[t2] : 0.0);
    if (top2) top2[r] = t2;
    if (cur_prob) {
      double c = 0.0;
      const bool masked = mask_state && mask_state[r] != 0;
      if (cur_tokens && !masked && cur_tokens[r] >= 0 && cur_tokens[r] < V) c = p[cur_tokens[r]];
      cur_prob[r] = c;
    }
  });
  return 0;
}

// Refresh rule (Sec. 4.2, Eq. archer-distance and Eq. archer-controller, with
// the cache-age signal A_t = t - r of Sec. 6 as an optional cap):
//   age_t = age[b] + 1                     (steps since the anchor, this one included)
//   D_t   = sum_i [g_cur[b,i] != g_anchor[b,i]]
//   flag  = D_t >= K  or  (max_age > 0 and age_t >= max_age)
// With update_anchor set, a flagged sequence takes g_anchor <- g_cur and
// age <- 0, an unflagged one age <- age_t; without it nothing is written
// except dist and flag.
int oracle_should_refresh(int B, int G, const int32_t* g_cur, int32_t* g_anchor, int32_t* age,
                          int K, int max_age, int update_anchor, int32_t* dist, uint8_t* flag) {
  if (B < 0 || G < 0) return -1;
  for (int b = 0; b < B; ++b) {
    int d = 0;
    for (int i = 0; i < G; ++i)
      if (g_cur[(size_t)b * G + i] != g_anchor[(size_t)b * G + i]) ++d;
    const int64_t age_t = (int64_t)age[b] + 1;
    const bool f = (d >= K) || (max_age > 0 && age_t >= max_age);
    dist[b] = d;
    flag[b] = f ? 1 : 0;
    if (update_anchor) {
      if (f) {
        for (int i = 0; i < G; ++i) g_anchor[(size_t)b * G + i] = g_cur[(size_t)b * G + i];
        age[b] = 0;
      } else {
        age[b] = (int32_t)age_t;
      }
    }
  }
  return 0;
}

int oracle_hardware_threads(void) { return (int)std::thread::hardware_concurrency(); }

}  // extern "C"
