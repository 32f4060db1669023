// Verify-step oracle: a plain, slow, fp64 CPU statement of what the verify step of
// lossless Psi-Spec decoding computes ("Unlocking Lossless Speedups in LLMs via
// Discrete Diffusion", Sec. 4.2 "One-step Diffusion w/ AR Verification" and
// Appendix B.3, Algorithm "Lossless Psi-Spec decoding (Linear Sampler)").
//
// TEST INFRASTRUCTURE ONLY. Nothing on the product path may link, load or call this
// file: only the tests, the package smoke check and the benchmark's CPU-baseline leg
// use it. It shares no code, header, table or helper with the CUDA library.
//
// Conventions (the readings of the paper are listed in the design notes):
//   * block size B is called gamma; the verify pass scores the block
//     [x^{L+1}, x~^1 .. x~^{B-1}] = block_tokens[0 .. gamma-1].
//   * target row j (0-based) is the verifier's distribution of block token j+1, so
//     the algorithm's p_i is target row i-1 and p_B (the bonus row) is row gamma-1.
//   * drafter row j is the distribution block token j was drawn from, so the
//     algorithm's q_i is drafter row i; drafter row 0 (q_0) is never read.
//   * uniforms[i-1] tests draft i (i = 1 .. gamma-1); uniforms[gamma-1] drives the
//     residual or bonus sample.
//   * temperature T > 0: p = softmax(l_target / T), q = softmax(l_drafter / T).
//     T == 0: greedy verification (accept iff the draft is the argmax of its target
//     row; correction and bonus are argmaxes; ties go to the lowest token id).
//   * filtered verification (the top-k / top-p sampling of the paper's evaluations,
//     Sec. 5.1, Sec. 5.2, Appendix C.1): p and q are replaced by their top-k, then
//     top-p filtered and renormalised forms p', q' before the same rule.
//
// Every floating-point step is fp64 on exactly decoded inputs; sums are plain
// left-to-right loops. Each function says which passage it follows.

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <thread>
#include <vector>

namespace {

// Input element decoding. dtype 0 = fp32, 1 = bf16 (the upper 16 bits of an fp32).
double load_elem(const void* base, int dtype, int64_t idx) {
  if (dtype == 0) {
    float f;
    std::memcpy(&f, static_cast<const char*>(base) + idx * 4, 4);
    return static_cast<double>(f);
  }
  uint16_t h;
  std::memcpy(&h, static_cast<const char*>(base) + idx * 2, 2);
  uint32_t bits = static_cast<uint32_t>(h) << 16;
  float f;
  std::memcpy(&f, &bits, 4);
  return static_cast<double>(f);
}

double bf16_bits_to_double(uint16_t h) {
  uint32_t bits = static_cast<uint32_t>(h) << 16;
  float f;
  std::memcpy(&f, &bits, 4);
  return static_cast<double>(f);
}

// Runs fn(i) for i in [0, n) on nthreads threads (0 = all hardware threads).
template <class F>
void parallel_for(int64_t n, int nthreads, F fn) {
  if (nthreads <= 0) nthreads = static_cast<int>(std::thread::hardware_concurrency());
  if (nthreads <= 1 || n <= 1) {
    for (int64_t i = 0; i < n; ++i) fn(i);
    return;
  }
  if (nthreads > n) nthreads = static_cast<int>(n);
  std::atomic<int64_t> next(0);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    pool.emplace_back([&]() {
      for (;;) {
        int64_t i = next.fetch_add(1);
        if (i >= n) break;
        fn(i);
      }
    });
  }
  for (auto& th : pool) th.join();
}

const double kInf = std::numeric_limits<double>::infinity();
const double kNaN = std::numeric_limits<double>::quiet_NaN();

}  // namespace

extern "C" {

// Number of hardware threads the oracle uses when asked for "all".
int oracle_hardware_threads(void) {
  return static_cast<int>(std::thread::hardware_concurrency());
}

// softmax(l / T) of one vocabulary row in fp64 (Sec. 4.2: the proposal and the
// verifier are categorical distributions given by softmax of the logits; Sec. 5.1
// "Setup": sampling temperature). z = l/T, m = max z, p = exp(z - m) / sum exp(z - m).
// Returns 0 on success, 1 if the row has no finite maximum or a non-finite sum
// (NaN or +inf logits, or every logit -inf).
int oracle_softmax(const double* logits, int64_t vocab, double temperature, double* p) {
  double m = -kInf;
  for (int64_t x = 0; x < vocab; ++x) {
    double z = logits[x] / temperature;
    if (std::isnan(z)) return 1;
    if (z > m) m = z;
  }
  if (!std::isfinite(m)) return 1;
  double s = 0.0;
  for (int64_t x = 0; x < vocab; ++x) {
    p[x] = std::exp(logits[x] / temperature - m);
    s += p[x];
  }
  if (!std::isfinite(s) || !(s > 0.0)) return 1;
  for (int64_t x = 0; x < vocab; ++x) p[x] /= s;
  return 0;
}

// Lowest index of the maximum of a row (greedy decoding at T = 0, Sec. 5.1:
// "temp=0 denotes greedy"; ties resolve to the lowest token id).
int64_t oracle_argmax(const double* row, int64_t vocab) {
  int64_t best = 0;
  for (int64_t x = 1; x < vocab; ++x)
    if (row[x] > row[best]) best = x;
  return best;
}

// Inverse-CDF draw from the unnormalised weights w (Alg. "Lossless Psi-Spec",
// the "sample" steps): the token is the smallest x with C(x) >= u * S, where
// C(x) = w(0) + ... + w(x) in ascending token order and S = C(V-1). If rounding
// leaves u*S above every C(x), the last token with positive weight is taken.
// *margin receives the distance, in the units of w, from u*S to the nearer of
// the two cumulative sums that bracket the chosen token.
int64_t oracle_inverse_cdf(const double* w, int64_t vocab, double u, double* margin) {
  double S = 0.0;
  for (int64_t x = 0; x < vocab; ++x) S += w[x];
  const double target = u * S;
  double C = 0.0;
  int64_t last_pos = -1;
  for (int64_t x = 0; x < vocab; ++x) {
    const double prev = C;
    C += w[x];
    if (w[x] > 0.0) last_pos = x;
    if (w[x] > 0.0 && C >= target) {
      if (margin) *margin = std::min(target - prev, C - target);
      return x;
    }
  }
  if (margin) *margin = 0.0;
  return last_pos;
}

// One verify decision for one sequence (Alg. "Lossless Psi-Spec decoding (Linear
// Sampler)", the steps after the verifier forward pass):
//   n = min({ i in [gamma-1] : r_i > min(1, p_i / q_i) } U { gamma }),
//   if n = gamma: sample from p_gamma (bonus), else from Norm([p_n - q_n]_+),
//   return [x^{L+1}, x~^{1:n-1}, z~].
// With the row conventions of this file, p_i = p_rows[i-1] and q_i = q_rows[i],
// both evaluated at the drafted token t_i (the algorithm writes them as scalars).
//
// p_rows, q_rows: [gamma][vocab] probability rows (greedy: raw scores whose argmax
// is taken; q_rows unused). tokens: [gamma]. uniforms: [gamma] in (0, 1].
// Outputs: *n_out = n; out_tokens[gamma+1] = emitted tokens, padded with -1;
// *num_emitted = n + 1; p_tok/q_tok[gamma] = p_i(t_i), q_i(t_i) (entry 0 is 0;
// entries after n are NaN); accept_margin[gamma] = |r_i - min(1, p_i/q_i)| for the
// decisions taken (entry 0 and entries after n are +inf; greedy: +inf);
// *sample_margin = the inverse-CDF margin of the final draw (greedy: +inf).
// Returns 0 on success, 2 if a token id is outside [0, vocab).
int oracle_accept_probs(int32_t gamma, int64_t vocab, const double* p_rows,
                        const double* q_rows, const int32_t* tokens,
                        const double* uniforms, int32_t greedy, int32_t* n_out,
                        int32_t* out_tokens, int32_t* num_emitted, double* p_tok,
                        double* q_tok, double* accept_margin, double* sample_margin) {
  for (int32_t i = 0; i < gamma; ++i)
    if (tokens[i] < 0 || tokens[i] >= vocab) return 2;
  for (int32_t i = 0; i < gamma; ++i) {
    p_tok[i] = (i == 0) ? 0.0 : kNaN;
    q_tok[i] = (i == 0) ? 0.0 : kNaN;
    accept_margin[i] = kInf;
  }
  int32_t n = gamma;
  for (int32_t i = 1; i < gamma; ++i) {
    const double* p_i = p_rows + static_cast<int64_t>(i - 1) * vocab;
    const int32_t t = tokens[i];
    if (greedy) {
      const int64_t a = oracle_argmax(p_i, vocab);
      p_tok[i] = (a == t) ? 1.0 : 0.0;
      q_tok[i] = 1.0;
      if (a != t) { n = i; break; }
      continue;
    }
    const double* q_i = q_rows + static_cast<int64_t>(i) * vocab;
    const double pv = p_i[t];
    const double qv = q_i[t];
    p_tok[i] = pv;
    q_tok[i] = qv;
    // q_i(t) = 0 cannot happen for a token drawn from q_i; if it does (underflow, or a
    // draft outside a filtered proposal's support), the ratio is +inf and the draft is
    // accepted when p_i(t) > 0, and 0 (rejected) when p_i(t) = 0 as well.
    const double ratio = (qv > 0.0) ? pv / qv : (pv > 0.0 ? kInf : 0.0);
    const double thresh = std::min(1.0, ratio);
    accept_margin[i] = std::fabs(uniforms[i - 1] - thresh);
    if (uniforms[i - 1] > thresh) { n = i; break; }
  }
  *n_out = n;

  // The final token: bonus from p_gamma (n == gamma) or the residual correction.
  int64_t z;
  const double u = uniforms[gamma - 1];
  const double* p_last = p_rows + static_cast<int64_t>(n - 1) * vocab;
  if (greedy) {
    z = oracle_argmax(p_last, vocab);
    *sample_margin = kInf;
  } else if (n == gamma) {
    z = oracle_inverse_cdf(p_last, vocab, u, sample_margin);
  } else {
    const double* q_n = q_rows + static_cast<int64_t>(n) * vocab;
    std::vector<double> w(static_cast<size_t>(vocab));
    double S = 0.0;
    for (int64_t x = 0; x < vocab; ++x) {
      w[x] = std::max(0.0, p_last[x] - q_n[x]);
      S += w[x];
    }
    // Norm([p_n - q_n]_+) is undefined when the residual has no mass; exact
    // arithmetic never rejects when p_n = q_n, so only rounding reaches this case,
    // and the draw falls back to p_n itself.
    if (S > 0.0)
      z = oracle_inverse_cdf(w.data(), vocab, u, sample_margin);
    else
      z = oracle_inverse_cdf(p_last, vocab, u, sample_margin);
  }

  for (int32_t k = 0; k <= gamma; ++k) out_tokens[k] = -1;
  for (int32_t k = 0; k < n; ++k) out_tokens[k] = tokens[k];
  out_tokens[n] = static_cast<int32_t>(z);
  *num_emitted = n + 1;
  return 0;
}

// oracle_accept_probs for `count` (tokens, uniforms) cases sharing one set of
// probability rows: tokens[count][gamma], uniforms[count][gamma]; outputs n_out[count],
// out_tokens[count][gamma+1], num_emitted[count]. Used to enumerate the rule's output
// distribution exactly. Returns the first nonzero per-case code, else 0.
int oracle_accept_probs_many(int64_t count, int32_t gamma, int64_t vocab, const double* p_rows,
                             const double* q_rows, const int32_t* tokens, const double* uniforms,
                             int32_t greedy, int32_t* n_out, int32_t* out_tokens,
                             int32_t* num_emitted, int32_t nthreads) {
  std::atomic<int> first_rc(0);
  parallel_for(count, nthreads, [&](int64_t c) {
    std::vector<double> ptok(gamma), qtok(gamma), am(gamma);
    double sm;
    int rc = oracle_accept_probs(gamma, vocab, p_rows, q_rows, tokens + c * gamma,
                                 uniforms + c * gamma, greedy, n_out + c,
                                 out_tokens + c * (gamma + 1), num_emitted + c, ptok.data(),
                                 qtok.data(), am.data(), &sm);
    if (rc) {
      int expected = 0;
      first_rc.compare_exchange_strong(expected, rc);
    }
  });
  return first_rc.load();
}

// The acceptance half of the verify step over a batch of sequences, from logits.
// target_logits, drafter_logits: [batch][gamma][vocab], dtype 0 = fp32, 1 = bf16.
// block_tokens: [batch][gamma]; temperature: [batch]; uniforms: [batch][gamma].
// Outputs per sequence b: num_accepted[b] = n - 1, out_tokens[b][gamma+1],
// num_emitted[b] = n + 1, diag[b][gamma][2] = (p_i(t_i), q_i(t_i)),
// accept_margin[b][gamma], sample_margin[b] (see oracle_accept_probs).
// A sequence with a token id outside [0, vocab) or a used row whose softmax is
// undefined gets num_accepted = -1, num_emitted = 0, out_tokens = -1 and a nonzero
// entry in status[b] (2 = token, 1 = logits); otherwise status[b] = 0.
// diag, accept_margin, sample_margin and status may be NULL.
int oracle_accept_block(int32_t batch, int32_t gamma, int64_t vocab, int32_t dtype,
                        const void* target_logits, const void* drafter_logits,
                        const int32_t* block_tokens, const float* temperature,
                        const float* uniforms, int32_t* num_accepted, int32_t* out_tokens,
                        int32_t* num_emitted, double* diag, double* accept_margin,
                        double* sample_margin, int32_t* status, int32_t nthreads) {
  if (batch < 0 || gamma < 1 || vocab < 1 || (dtype != 0 && dtype != 1)) return -1;
  parallel_for(batch, nthreads, [&](int64_t b) {
    const int64_t row0 = b * gamma;
    const double T = static_cast<double>(temperature[b]);
    const bool greedy = !(T > 0.0);
    std::vector<double> p_rows(static_cast<size_t>(gamma) * vocab);
    std::vector<double> q_rows(greedy ? 0 : static_cast<size_t>(gamma) * vocab);
    std::vector<double> raw(static_cast<size_t>(vocab));
    int bad = 0;
    for (int32_t j = 0; j < gamma && !bad; ++j) {
      for (int64_t x = 0; x < vocab; ++x)
        raw[x] = load_elem(target_logits, dtype, (row0 + j) * vocab + x);
      if (greedy) {
        for (int64_t x = 0; x < vocab; ++x) {
          if (std::isnan(raw[x])) bad = 1;
          p_rows[j * vocab + x] = raw[x];
        }
      } else {
        bad |= oracle_softmax(raw.data(), vocab, T, &p_rows[j * vocab]);
      }
    }
    if (!greedy) {
      for (int32_t j = 1; j < gamma && !bad; ++j) {
        for (int64_t x = 0; x < vocab; ++x)
          raw[x] = load_elem(drafter_logits, dtype, (row0 + j) * vocab + x);
        bad |= oracle_softmax(raw.data(), vocab, T, &q_rows[j * vocab]);
      }
    }
    std::vector<double> u(static_cast<size_t>(gamma));
    for (int32_t j = 0; j < gamma; ++j) u[j] = static_cast<double>(uniforms[row0 + j]);
    std::vector<double> ptok(gamma), qtok(gamma), am(gamma);
    double sm = kInf;
    int32_t n = 0, ne = 0;
    int32_t* ot = out_tokens + b * (gamma + 1);
    int rc = 0;
    for (int32_t j = 0; j < gamma; ++j)
      if (block_tokens[row0 + j] < 0 || block_tokens[row0 + j] >= vocab) rc = 2;
    if (rc == 0 && !bad)
      rc = oracle_accept_probs(gamma, vocab, p_rows.data(), greedy ? nullptr : q_rows.data(),
                               block_tokens + row0, u.data(), greedy ? 1 : 0, &n, ot, &ne,
                               ptok.data(), qtok.data(), am.data(), &sm);
    const int code = rc ? rc : (bad ? 1 : 0);
    if (status) status[b] = code;
    if (code) {
      num_accepted[b] = -1;
      num_emitted[b] = 0;
      for (int32_t k = 0; k <= gamma; ++k) ot[k] = -1;
      for (int32_t j = 0; j < gamma; ++j) { ptok[j] = kNaN; qtok[j] = kNaN; am[j] = kInf; }
      sm = kInf;
    } else {
      num_accepted[b] = n - 1;
      num_emitted[b] = ne;
    }
    for (int32_t j = 0; j < gamma; ++j) {
      if (diag) {
        diag[(row0 + j) * 2 + 0] = ptok[j];
        diag[(row0 + j) * 2 + 1] = qtok[j];
      }
      if (accept_margin) accept_margin[row0 + j] = am[j];
    }
    if (sample_margin) sample_margin[b] = sm;
  });
  return 0;
}

// Top-k / top-p filtering of one probability row (the paper decodes with top-k 50
// and top-p 0.95, Sec. 5.1, Sec. 5.2 and Appendix C.1; the order of the two filters is
// not stated, and the common one is taken): tokens are ranked by probability, ties
// to the lower token id; the first top_k are kept; of those, renormalised, the
// shortest prefix in rank order whose mass reaches top_p is kept; the kept
// probabilities are renormalised to sum to 1 and every other token gets 0.
// out[vocab] receives the filtered row. *margin (may be NULL) receives the distance
// from top_p to the nearer of the two renormalised cumulative masses that bracket
// the cut (+inf when the cut is set by top_k alone). Returns 0, or 1 if top_k < 1 or
// top_p is outside (0, 1].
int oracle_filter_row(const double* p, int64_t vocab, int32_t top_k, double top_p, double* out,
                      double* margin) {
  if (top_k < 1 || !(top_p > 0.0) || top_p > 1.0) return 1;
  std::vector<int64_t> order(static_cast<size_t>(vocab));
  for (int64_t x = 0; x < vocab; ++x) order[x] = x;
  std::stable_sort(order.begin(), order.end(),
                   [&](int64_t a, int64_t b) { return p[a] > p[b]; });
  const int64_t k = std::min<int64_t>(top_k, vocab);
  double mass_k = 0.0;
  for (int64_t j = 0; j < k; ++j) mass_k += p[order[j]];
  // shortest prefix of the top-k, renormalised, whose mass reaches top_p (top_p = 1
  // keeps the whole top-k: no rounding of the running sum may cut its tail)
  int64_t keep = k;
  double m = kInf, c = 0.0;
  for (int64_t j = 0; j < k && top_p < 1.0; ++j) {
    const double before = c;
    c += p[order[j]] / mass_k;
    if (c >= top_p) {
      keep = j + 1;
      m = std::min(top_p - before, c - top_p);
      break;
    }
  }
  if (margin) *margin = m;
  double kept = 0.0;
  for (int64_t j = 0; j < keep; ++j) kept += p[order[j]];
  for (int64_t x = 0; x < vocab; ++x) out[x] = 0.0;
  for (int64_t j = 0; j < keep; ++j) out[order[j]] = p[order[j]] / kept;
  return 0;
}

// oracle_accept_block with top-k / top-p filtering of both the target and the drafter
// distributions (oracle_filter_row with the sequence's top_k[b], top_p[b]) before the
// decisions and the final draw; greedy sequences (T = 0) are unchanged, since the
// filter always keeps the argmax. filter_margin[b] (may be NULL) receives the smallest
// top-p margin over the rows the sequence uses. A top_k or top_p outside its range
// counts as bad input (status 3).
int oracle_accept_block_filtered(int32_t batch, int32_t gamma, int64_t vocab, int32_t dtype,
                                 const void* target_logits, const void* drafter_logits,
                                 const int32_t* block_tokens, const float* temperature,
                                 const int32_t* top_k, const float* top_p, const float* uniforms,
                                 int32_t* num_accepted, int32_t* out_tokens,
                                 int32_t* num_emitted, double* diag, double* accept_margin,
                                 double* sample_margin, double* filter_margin, int32_t* status,
                                 int32_t nthreads) {
  if (batch < 0 || gamma < 1 || vocab < 1 || (dtype != 0 && dtype != 1)) return -1;
  parallel_for(batch, nthreads, [&](int64_t b) {
    const int64_t row0 = b * gamma;
    const double T = static_cast<double>(temperature[b]);
    const bool greedy = !(T > 0.0);
    const int32_t k = top_k[b];
    const double tp = static_cast<double>(top_p[b]);
    std::vector<double> p_rows(static_cast<size_t>(gamma) * vocab);
    std::vector<double> q_rows(greedy ? 0 : static_cast<size_t>(gamma) * vocab);
    std::vector<double> raw(static_cast<size_t>(vocab)), sm_row(static_cast<size_t>(vocab));
    int bad = 0, badf = 0;
    double fm = kInf;
    if (k < 1 || !(tp > 0.0) || tp > 1.0) badf = 1;
    for (int32_t j = 0; j < gamma && !bad; ++j) {
      for (int64_t x = 0; x < vocab; ++x)
        raw[x] = load_elem(target_logits, dtype, (row0 + j) * vocab + x);
      if (greedy) {
        for (int64_t x = 0; x < vocab; ++x) {
          if (std::isnan(raw[x])) bad = 1;
          p_rows[j * vocab + x] = raw[x];
        }
      } else {
        bad |= oracle_softmax(raw.data(), vocab, T, sm_row.data());
        double m = kInf;
        if (!bad && !badf) {
          oracle_filter_row(sm_row.data(), vocab, k, tp, &p_rows[j * vocab], &m);
          fm = std::min(fm, m);
        }
      }
    }
    if (!greedy) {
      for (int32_t j = 1; j < gamma && !bad; ++j) {
        for (int64_t x = 0; x < vocab; ++x)
          raw[x] = load_elem(drafter_logits, dtype, (row0 + j) * vocab + x);
        bad |= oracle_softmax(raw.data(), vocab, T, sm_row.data());
        double m = kInf;
        if (!bad && !badf) {
          oracle_filter_row(sm_row.data(), vocab, k, tp, &q_rows[j * vocab], &m);
          fm = std::min(fm, m);
        }
      }
    }
    std::vector<double> u(static_cast<size_t>(gamma));
    for (int32_t j = 0; j < gamma; ++j) u[j] = static_cast<double>(uniforms[row0 + j]);
    std::vector<double> ptok(gamma), qtok(gamma), am(gamma);
    double sm = kInf;
    int32_t n = 0, ne = 0;
    int32_t* ot = out_tokens + b * (gamma + 1);
    int rc = 0;
    for (int32_t j = 0; j < gamma; ++j)
      if (block_tokens[row0 + j] < 0 || block_tokens[row0 + j] >= vocab) rc = 2;
    if (rc == 0 && !bad && !(badf && !greedy))
      rc = oracle_accept_probs(gamma, vocab, p_rows.data(), greedy ? nullptr : q_rows.data(),
                               block_tokens + row0, u.data(), greedy ? 1 : 0, &n, ot, &ne,
                               ptok.data(), qtok.data(), am.data(), &sm);
    const int code = rc ? rc : (bad ? 1 : ((badf && !greedy) ? 3 : 0));
    if (status) status[b] = code;
    if (code) {
      num_accepted[b] = -1;
      num_emitted[b] = 0;
      for (int32_t kk = 0; kk <= gamma; ++kk) ot[kk] = -1;
      for (int32_t j = 0; j < gamma; ++j) { ptok[j] = kNaN; qtok[j] = kNaN; am[j] = kInf; }
      sm = kInf;
      fm = kInf;
    } else {
      num_accepted[b] = n - 1;
      num_emitted[b] = ne;
    }
    for (int32_t j = 0; j < gamma; ++j) {
      if (diag) {
        diag[(row0 + j) * 2 + 0] = ptok[j];
        diag[(row0 + j) * 2 + 1] = qtok[j];
      }
      if (accept_margin) accept_margin[row0 + j] = am[j];
    }
    if (sample_margin) sample_margin[b] = sm;
    if (filter_margin) filter_margin[b] = greedy ? kInf : fm;
  });
  return 0;
}

// Draft-side sampling (Alg. "Lossless Psi-Spec decoding (Linear Sampler)": the free
// clean token x^{L+1} ~ q_0 and the B-1 drafts x~ ~ q, sampled in parallel). Drafter
// row j of sequence b (q_0 for j = 0, the diffusion rows after it) is softmaxed at the
// sequence's temperature, top-k / top-p filtered when top_k is not NULL (as in
// oracle_accept_block_filtered), and block token j is the inverse-CDF draw with
// uniforms[b][j] in ascending token order. At T = 0 it is the row's lowest-index argmax.
// Outputs per (b, j): tokens, q_tok (the drawn token's probability; 1 at T = 0), margin
// (the inverse-CDF margin; +inf at T = 0), filter_margin (the top-p margin; +inf
// unfiltered or at T = 0). status[b]: 0, 1 (NaN or undefined softmax in a row), 3 (a
// tempered sequence's top_k / top_p out of range); a flagged sequence's tokens are -1.
int oracle_sample_block(int32_t batch, int32_t gamma, int64_t vocab, int32_t dtype,
                        const void* drafter_logits, const float* temperature,
                        const int32_t* top_k, const float* top_p, const float* uniforms,
                        int32_t* tokens, double* q_tok, double* margin, double* filter_margin,
                        int32_t* status, int32_t nthreads) {
  if (batch < 0 || gamma < 1 || vocab < 1 || (dtype != 0 && dtype != 1)) return -1;
  parallel_for(batch, nthreads, [&](int64_t b) {
    const double T = static_cast<double>(temperature[b]);
    const bool greedy = !(T > 0.0);
    const bool filtered = top_k != nullptr && !greedy;
    int code = 0;
    if (filtered && (top_k[b] < 1 || !(top_p[b] > 0.0f) || top_p[b] > 1.0f)) code = 3;
    std::vector<double> raw(static_cast<size_t>(vocab)), q(static_cast<size_t>(vocab)),
        qf(static_cast<size_t>(vocab));
    std::vector<int32_t> tok(gamma, -1);
    std::vector<double> qt(gamma, kNaN), mg(gamma, kInf), fm(gamma, kInf);
    for (int32_t j = 0; j < gamma && code == 0; ++j) {
      const int64_t row = b * gamma + j;
      for (int64_t x = 0; x < vocab; ++x) raw[x] = load_elem(drafter_logits, dtype, row * vocab + x);
      if (greedy) {
        for (int64_t x = 0; x < vocab; ++x)
          if (std::isnan(raw[x])) code = 1;
        if (code) break;
        tok[j] = static_cast<int32_t>(oracle_argmax(raw.data(), vocab));
        qt[j] = 1.0;
        continue;
      }
      if (oracle_softmax(raw.data(), vocab, T, q.data())) { code = 1; break; }
      const double* w = q.data();
      if (filtered) {
        oracle_filter_row(q.data(), vocab, top_k[b], static_cast<double>(top_p[b]), qf.data(),
                          &fm[j]);
        w = qf.data();
      }
      const double u = static_cast<double>(uniforms[row]);
      const int64_t x = oracle_inverse_cdf(w, vocab, u, &mg[j]);
      tok[j] = static_cast<int32_t>(x);
      qt[j] = w[x];
    }
    status[b] = code;
    for (int32_t j = 0; j < gamma; ++j) {
      const int64_t row = b * gamma + j;
      tokens[row] = code ? -1 : tok[j];
      if (q_tok) q_tok[row] = code ? kNaN : qt[j];
      if (margin) margin[row] = code ? kInf : mg[j];
      if (filter_margin) filter_margin[row] = code ? kInf : fm[j];
    }
  });
  return 0;
}

// Block-causal verify attention over a paged KV cache with grouped-query heads
// (Sec. 4.1: the block is scored while the prefix activations stay in the KV
// cache; Alg. "Lossless Psi-Spec": p <- x_theta([x^{L+1}, x~]; x) is one causal
// forward pass over the block). For sequence b with kv_len[b] keys, the block's
// own keys sit at positions ctx = kv_len[b] - gamma .. kv_len[b] - 1, and block
// query j attends to every key k <= ctx + j. Query head h reads KV head
// h / (num_q_heads / num_kv_heads). Logical key k lives in physical page
// page_table[b][k / page_size], slot k % page_size.
// q: bf16 [batch][gamma][Hq][D]; k_cache, v_cache: bf16 [num_pages][Hkv][page_size][D];
// out: fp64 [batch][gamma][Hq][D]; lse: fp64 [batch][gamma][Hq] (natural log of the
// softmax normaliser of the scaled scores), may be NULL.
// rows: optional list of nrows (b, j, h) triples to compute (NULL = all rows).
// A sequence whose kv_len is outside [gamma, max_pages * page_size] or that maps a
// visible key to a page id outside [0, num_pages) gets out = 0, lse = -inf and
// status[b] = 1 (status may be NULL).
//
// tree_mask (may be NULL): [batch][gamma] bit sets for tree verification (Sec. 4.2:
// several candidates verified in one pass as a prefix tree). Block query j then sees the prefix keys k < ctx and the block keys
// ctx + i for every bit i set in tree_mask[b][j] (its ancestors and itself), instead
// of every k <= ctx + j. gamma <= 64 with a mask.
int oracle_verify_attention_tree(int32_t batch, int32_t gamma, int32_t num_q_heads,
                                 int32_t num_kv_heads, int32_t head_dim, int32_t page_size,
                                 int32_t max_pages_per_seq, int32_t num_pages,
                                 double softmax_scale, const uint16_t* q, const uint16_t* k_cache,
                                 const uint16_t* v_cache, const int32_t* page_table,
                                 const int32_t* kv_len, const uint64_t* tree_mask, double* out,
                                 double* lse, const int32_t* rows, int64_t nrows, int32_t* status,
                                 int32_t nthreads) {
  if (tree_mask && gamma > 64) return -1;
  if (batch < 0 || gamma < 1 || num_q_heads < 1 || num_kv_heads < 1 ||
      num_q_heads % num_kv_heads != 0 || head_dim < 1 || page_size < 1)
    return -1;
  const int32_t group = num_q_heads / num_kv_heads;
  const int32_t D = head_dim;
  std::vector<int32_t> seq_bad(static_cast<size_t>(batch), 0);
  for (int32_t b = 0; b < batch; ++b) {
    const int32_t L = kv_len[b];
    if (L < gamma || static_cast<int64_t>(L) > static_cast<int64_t>(max_pages_per_seq) * page_size) {
      seq_bad[b] = 1;
      continue;
    }
    const int32_t used_pages = (L + page_size - 1) / page_size;
    for (int32_t i = 0; i < used_pages; ++i) {
      const int32_t pg = page_table[static_cast<int64_t>(b) * max_pages_per_seq + i];
      if (pg < 0 || pg >= num_pages) seq_bad[b] = 1;
    }
  }
  if (status)
    for (int32_t b = 0; b < batch; ++b) status[b] = seq_bad[b];
  const int64_t total = rows ? nrows : static_cast<int64_t>(batch) * gamma * num_q_heads;
  parallel_for(total, nthreads, [&](int64_t idx) {
    int32_t b, j, h;
    if (rows) {
      b = rows[idx * 3 + 0]; j = rows[idx * 3 + 1]; h = rows[idx * 3 + 2];
    } else {
      h = static_cast<int32_t>(idx % num_q_heads);
      j = static_cast<int32_t>((idx / num_q_heads) % gamma);
      b = static_cast<int32_t>(idx / (static_cast<int64_t>(num_q_heads) * gamma));
    }
    const int64_t orow = (static_cast<int64_t>(b) * gamma + j) * num_q_heads + h;
    double* o = out + orow * D;
    if (seq_bad[b]) {
      for (int32_t d = 0; d < D; ++d) o[d] = 0.0;
      if (lse) lse[orow] = -kInf;
      return;
    }
    const int32_t g = h / group;
    const int32_t ctx = kv_len[b] - gamma;
    // the visible keys, in increasing order
    std::vector<int32_t> vis;
    for (int32_t k = 0; k < ctx; ++k) vis.push_back(k);
    for (int32_t i = 0; i < gamma; ++i) {
      const bool seen = tree_mask ? ((tree_mask[static_cast<int64_t>(b) * gamma + j] >> i) & 1u) != 0
                                  : i <= j;
      if (seen) vis.push_back(ctx + i);
    }
    const int32_t nvis = static_cast<int32_t>(vis.size());
    std::vector<double> qv(D), s(nvis);
    for (int32_t d = 0; d < D; ++d) qv[d] = bf16_bits_to_double(q[orow * D + d]);
    auto kv_offset = [&](int32_t k) {
      const int32_t pg = page_table[static_cast<int64_t>(b) * max_pages_per_seq + k / page_size];
      return ((static_cast<int64_t>(pg) * num_kv_heads + g) * page_size + k % page_size) * D;
    };
    double m = -kInf;
    for (int32_t k = 0; k < nvis; ++k) {
      const int64_t off = kv_offset(vis[k]);
      double dot = 0.0;
      for (int32_t d = 0; d < D; ++d) dot += qv[d] * bf16_bits_to_double(k_cache[off + d]);
      s[k] = dot * softmax_scale;
      if (s[k] > m) m = s[k];
    }
    double l = 0.0;
    for (int32_t k = 0; k < nvis; ++k) {
      s[k] = std::exp(s[k] - m);
      l += s[k];
    }
    std::vector<double> acc(D, 0.0);  // local: a row listed twice is computed twice
    for (int32_t k = 0; k < nvis; ++k) {
      const int64_t off = kv_offset(vis[k]);
      const double pk = s[k] / l;
      for (int32_t d = 0; d < D; ++d) acc[d] += pk * bf16_bits_to_double(v_cache[off + d]);
    }
    for (int32_t d = 0; d < D; ++d) o[d] = acc[d];
    if (lse) lse[orow] = m + std::log(l);
  });
  return 0;
}

int oracle_verify_attention(int32_t batch, int32_t gamma, int32_t num_q_heads,
                            int32_t num_kv_heads, int32_t head_dim, int32_t page_size,
                            int32_t max_pages_per_seq, int32_t num_pages, double softmax_scale,
                            const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache,
                            const int32_t* page_table, const int32_t* kv_len, double* out,
                            double* lse, const int32_t* rows, int64_t nrows, int32_t* status,
                            int32_t nthreads) {
  return oracle_verify_attention_tree(batch, gamma, num_q_heads, num_kv_heads, head_dim,
                                      page_size, max_pages_per_seq, num_pages, softmax_scale, q,
                                      k_cache, v_cache, page_table, kv_len, nullptr, out, lse,
                                      rows, nrows, status, nthreads);
}

}  // extern "C"
