// nmv_sweep.cu -- the full-coverage escalation harness (nmv_sweep): the
// engine's validation escalation (Section 4.3, "Full-coverage evaluation";
// Figure 3, bottom-right; S6.1): a lightweight case set is validated first,
// and only when every one of its cases passes does the extended set (all
// shapes and dtypes) run.  Each set is one nmv_validate_batch call (one scan
// launch per element type, one finalize).  The per-case pass/fail and match
// rates are written as a canonical text record and sealed with its SHA-256
// digest, so the evidence behind an acceptance cannot change unnoticed.
//
// SHA-256 follows FIPS 180-4; its round constants and initial hash value
// (the first 32 fractional bits of the cube roots of the first 64 primes and
// of the square roots of the first 8) are derived here with exact integer
// roots, not typed in.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "nmv_internal.h"

namespace nmv {
namespace {

// ---------------------------------------------------------------- SHA-256
typedef unsigned __int128 u128;

// floor(x^(1/k)) of a 128-bit x (k = 2 or 3), by bisection on the integers.
uint64_t iroot(u128 x, int k) {
  uint64_t lo = 0, hi = 1ull << 43;  // (2^43)^3 > 2^105 > every x used here
  while (lo < hi) {
    const uint64_t mid = lo + (hi - lo + 1) / 2;
    u128 p = (u128)mid * mid;
    if (k == 3) p *= mid;
    if (p <= x) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

struct ShaConst {
  uint32_t k[64];
  uint32_t h0[8];
  ShaConst() {
    int primes[64], n = 0;
    for (int c = 2; n < 64; ++c) {
      bool prime = true;
      for (int d = 2; d * d <= c; ++d)
        if (c % d == 0) prime = false;
      if (prime) primes[n++] = c;
    }
    // first 32 fractional bits of p^(1/3): the low 32 bits of
    // floor(p^(1/3) * 2^32) = floor((p * 2^96)^(1/3)); of p^(1/2) likewise
    for (int i = 0; i < 64; ++i) k[i] = (uint32_t)iroot((u128)primes[i] << 96, 3);
    for (int i = 0; i < 8; ++i) h0[i] = (uint32_t)iroot((u128)primes[i] << 64, 2);
  }
};

const ShaConst &sha_const() {
  static const ShaConst c;
  return c;
}

inline uint32_t rotr(uint32_t x, int n) { return (x >> n) | (x << (32 - n)); }

void sha256(const uint8_t *msg, size_t len, uint8_t out[32]) {
  const ShaConst &C = sha_const();
  uint32_t h[8];
  std::memcpy(h, C.h0, sizeof h);
  // padding: 0x80, zeros, the bit length as a 64-bit big-endian integer
  std::vector<uint8_t> m(msg, msg + len);
  m.push_back(0x80);
  while (m.size() % 64 != 56) m.push_back(0);
  const uint64_t bits = (uint64_t)len * 8;
  for (int i = 7; i >= 0; --i) m.push_back((uint8_t)(bits >> (8 * i)));
  for (size_t blk = 0; blk < m.size(); blk += 64) {
    uint32_t w[64];
    for (int t = 0; t < 16; ++t)
      w[t] = (uint32_t)m[blk + 4 * t] << 24 | (uint32_t)m[blk + 4 * t + 1] << 16 | (uint32_t)m[blk + 4 * t + 2] << 8 |
             (uint32_t)m[blk + 4 * t + 3];
    for (int t = 16; t < 64; ++t) {
      const uint32_t s0 = rotr(w[t - 15], 7) ^ rotr(w[t - 15], 18) ^ (w[t - 15] >> 3);
      const uint32_t s1 = rotr(w[t - 2], 17) ^ rotr(w[t - 2], 19) ^ (w[t - 2] >> 10);
      w[t] = w[t - 16] + s0 + w[t - 7] + s1;
    }
    uint32_t a = h[0], b = h[1], c = h[2], d = h[3], e = h[4], f = h[5], g = h[6], hh = h[7];
    for (int t = 0; t < 64; ++t) {
      const uint32_t S1 = rotr(e, 6) ^ rotr(e, 11) ^ rotr(e, 25);
      const uint32_t ch = (e & f) ^ (~e & g);
      const uint32_t t1 = hh + S1 + ch + C.k[t] + w[t];
      const uint32_t S0 = rotr(a, 2) ^ rotr(a, 13) ^ rotr(a, 22);
      const uint32_t maj = (a & b) ^ (a & c) ^ (b & c);
      const uint32_t t2 = S0 + maj;
      hh = g;
      g = f;
      f = e;
      e = d + t1;
      d = c;
      c = b;
      b = a;
      a = t1 + t2;
    }
    h[0] += a;
    h[1] += b;
    h[2] += c;
    h[3] += d;
    h[4] += e;
    h[5] += f;
    h[6] += g;
    h[7] += hh;
  }
  for (int i = 0; i < 8; ++i)
    for (int j = 0; j < 4; ++j) out[4 * i + j] = (uint8_t)(h[i] >> (24 - 8 * j));
}

// ------------------------------------------------------------ the sweep
// A case raises an integrity hazard when its candidate passes an input
// through, or is constant or all zero while the reference is not.
bool hazard(uint32_t f) {
  if (f & NMV_FLAG_CAND_EQ_INPUT) return true;
  if ((f & NMV_FLAG_CAND_CONSTANT) && !(f & NMV_FLAG_REF_CONSTANT)) return true;
  if ((f & NMV_FLAG_CAND_ALL_ZERO) && !(f & NMV_FLAG_REF_ALL_ZERO)) return true;
  return false;
}

void append(std::string &s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
void append(std::string &s, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  const int n = std::vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  s.append(buf, (size_t)std::min(n, (int)sizeof buf - 1));
}

}  // namespace
}  // namespace nmv

extern "C" int nmv_validate_batch(const nmv_case *cases, int64_t n, void *cuda_stream, nmv_result **out);
extern "C" void nmv_result_free(void *r);

namespace nmv {
namespace {

int run_sweep(const nmv_case *light, int64_t n_light, const nmv_case *ext, int64_t n_ext, void *stream,
              nmv_sweep_report **out) {
  if (out == nullptr) return host_fail(NMV_EINVAL, "out is NULL");
  *out = nullptr;
  if (n_light < 1 || n_light > NMV_MAX_CASES || light == nullptr)
    return host_fail(NMV_EINVAL, "the lightweight set needs 1 .. NMV_MAX_CASES cases");
  if (n_ext < 0 || n_ext > NMV_MAX_CASES || (n_ext > 0 && ext == nullptr))
    return host_fail(NMV_EINVAL, "the extended set needs 0 .. NMV_MAX_CASES cases");
  nmv_result *rl = nullptr, *re = nullptr;
  int rc = nmv_validate_batch(light, n_light, stream, &rl);
  if (rc) {
    const std::string msg = std::string("lightweight set: ") + nmv_last_error();
    return host_fail(rc, msg);
  }
  struct Free {
    nmv_result *&p;
    ~Free() {
      if (p) nmv_result_free(p);
    }
  } fl{rl}, fe{re};
  int64_t pass_l = 0;
  uint32_t fany = 0;
  bool haz = false;
  for (int64_t i = 0; i < n_light; ++i) {
    pass_l += rl[i].pass;
    fany |= rl[i].flags;
    haz = haz || hazard(rl[i].flags);
  }
  const bool escalate = pass_l == n_light && n_ext > 0;
  int64_t pass_e = 0;
  if (escalate) {
    rc = nmv_validate_batch(ext, n_ext, stream, &re);
    if (rc) {
      const std::string msg = std::string("extended set: ") + nmv_last_error();
      return host_fail(rc, msg);
    }
    for (int64_t i = 0; i < n_ext; ++i) {
      pass_e += re[i].pass;
      fany |= re[i].flags;
      haz = haz || hazard(re[i].flags);
    }
  }
  const int64_t n_run = n_light + (escalate ? n_ext : 0);
  const bool accepted = pass_l == n_light && (n_ext == 0 || (escalate && pass_e == n_ext)) && !haz;

  // the evidence record: one header line, one line per validated case
  std::string ev;
  append(ev, "nmv-sweep v1 light=%lld ext=%lld escalated=%d accepted=%d pass_light=%lld pass_ext=%lld\n",
         (long long)n_light, (long long)n_ext, escalate ? 1 : 0, accepted ? 1 : 0, (long long)pass_l,
         (long long)pass_e);
  auto line = [&](const char *set, int64_t i, const nmv_result &r, const nmv_case &c) {
    append(ev, "%s %lld dtype=%d numel=%lld pass=%d mismatch=%lld match=%.17g max_abs=%.17g max_rel=%.17g "
               "nonfinite=%lld flags=%u\n",
           set, (long long)i, c.cand.dtype, (long long)r.numel, r.pass, (long long)r.mismatch, r.match_fraction,
           r.max_abs, r.max_rel,
           (long long)(r.cand_nan + r.cand_posinf + r.cand_neginf + r.ref_nan + r.ref_posinf + r.ref_neginf),
           r.flags);
  };
  for (int64_t i = 0; i < n_light; ++i) line("L", i, rl[i], light[i]);
  if (escalate)
    for (int64_t i = 0; i < n_ext; ++i) line("E", i, re[i], ext[i]);

  // the report, its evidence text and a copy of every result record (the
  // record arrays stay in the validate result blocks, kept until the report
  // is released)
  const size_t rep = (sizeof(nmv_sweep_report) + 15) / 16 * 16;
  const size_t res = (sizeof(nmv_result) * (size_t)n_run + 15) / 16 * 16;
  uint8_t *blk = (uint8_t *)std::calloc(1, rep + res + ev.size() + 1);
  if (!blk) return host_fail(NMV_ENOMEM, "report allocation");
  nmv_sweep_report *R = (nmv_sweep_report *)blk;
  R->status = NMV_OK;
  R->escalated = escalate ? 1 : 0;
  R->accepted = accepted ? 1 : 0;
  R->n_light = n_light;
  R->n_ext = n_ext;
  R->n_run = n_run;
  R->n_pass_light = pass_l;
  R->n_pass_ext = pass_e;
  R->match_rate_light = (double)pass_l / (double)n_light;
  R->match_rate_ext = escalate ? (double)pass_e / (double)n_ext : 0.0;
  R->flags_any = fany;
  R->results = (nmv_result *)(blk + rep);
  std::memcpy(R->results, rl, sizeof(nmv_result) * (size_t)n_light);
  if (escalate) std::memcpy(R->results + n_light, re, sizeof(nmv_result) * (size_t)n_ext);
  R->evidence = (char *)(blk + rep + res);
  std::memcpy(R->evidence, ev.data(), ev.size());
  R->evidence_len = (int64_t)ev.size();
  sha256((const uint8_t *)ev.data(), ev.size(), R->digest);
  R->blocks[0] = rl;
  R->blocks[1] = re;
  rl = re = nullptr;  // owned by the report now
  *out = R;
  host_clear_error();
  return NMV_OK;
}

}  // namespace
}  // namespace nmv

extern "C" int nmv_sweep(const nmv_case *light, int64_t n_light, const nmv_case *ext, int64_t n_ext,
                         void *cuda_stream, nmv_sweep_report **out) {
  return nmv::run_sweep(light, n_light, ext, n_ext, cuda_stream, out);
}

extern "C" void nmv_sweep_free(nmv_sweep_report *r) {
  if (!r) return;
  if (r->blocks[0]) nmv_result_free(r->blocks[0]);
  if (r->blocks[1]) nmv_result_free(r->blocks[1]);
  std::free(r);
}

extern "C" void nmv_sha256(const void *data, int64_t len, uint8_t out[32]) {
  nmv::sha256((const uint8_t *)data, len > 0 ? (size_t)len : 0, out);
}
