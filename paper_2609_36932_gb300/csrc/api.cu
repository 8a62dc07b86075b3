// Host-side parts of libfastrl_grpo: error reporting, the launch counter, the workspace protocol
// and adaptive rollout sampling (Sec. 3.3, Eqs. 10-14; Algorithm 1 Phases 1a and 1b).
#define GRPO_TU 8  // this file's bit in the checked build's report (grpo_debug_checks)
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "common.cuh"

namespace fastrl {

namespace {
thread_local char g_msg[512] = {0};
std::atomic<uint64_t> g_launches{0};
}  // namespace

grpo_status fail(grpo_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof g_msg, fmt, ap);
  va_end(ap);
  return s;
}

void clear_error() { g_msg[0] = 0; }

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

// Test hook (grpo_test_fail_launch): the n-th next launch check reports a failure.
std::atomic<int> g_fail_countdown{0};

grpo_status check_launch(const char* what) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  if (g_fail_countdown.load(std::memory_order_relaxed) > 0 &&
      g_fail_countdown.fetch_sub(1, std::memory_order_relaxed) == 1)
    return fail(GRPO_ERR_CUDA, "%s: injected launch failure (grpo_test_fail_launch)", what);
  return GRPO_OK;
}

grpo_status workspace_check(void* ws, size_t* ws_bytes, size_t need, const char* who,
                            bool* query_only) {
  *query_only = false;
  if (ws == nullptr) {
    if (ws_bytes == nullptr) {
      if (need == 0) return GRPO_OK;
      return fail(GRPO_ERR_WORKSPACE, "%s: needs %zu workspace bytes but ws and ws_bytes are NULL",
                  who, need);
    }
    *ws_bytes = need;
    *query_only = true;
    return GRPO_OK;
  }
  if (ws_bytes == nullptr || *ws_bytes < need)
    return fail(GRPO_ERR_WORKSPACE, "%s: workspace of %zu bytes given, %zu needed", who,
                ws_bytes ? *ws_bytes : (size_t)0, need);
  if (reinterpret_cast<uintptr_t>(ws) % 256 != 0)
    return fail(GRPO_ERR_WORKSPACE, "%s: workspace must be 256-byte aligned", who);
  return GRPO_OK;
}

}  // namespace fastrl

using namespace fastrl;

extern "C" const char* grpo_last_error(void) { return g_msg; }

#if defined(GRPO_CHECKED)
extern "C" const char* grpo_version(void) { return "fastrl_grpo 0.1.0 (sm_103a, checked)"; }
#else
extern "C" const char* grpo_version(void) { return "fastrl_grpo 0.1.0 (sm_103a)"; }
#endif

extern "C" grpo_status grpo_debug_checks(int32_t reset, int32_t* file_mask, int32_t* first_site) {
  clear_error();
  if (!file_mask || !first_site)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_debug_checks: NULL output");
  *file_mask = 0;
  *first_site = 0;
#if defined(GRPO_CHECKED)
  const cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess)
    return fail(GRPO_ERR_CUDA, "grpo_debug_checks: cudaDeviceSynchronize: %s", cudaGetErrorString(e));
  grpo_status (*const readers[])(bool, int32_t*, int32_t*) = {
      dcheck_read_advantage, dcheck_read_prune, dcheck_read_compact, dcheck_read_loss,
      dcheck_read_gspo,      dcheck_read_reduce, dcheck_read_lmhead, dcheck_read_gemm};
  for (auto rd : readers)
    if (rd(reset != 0, file_mask, first_site) != GRPO_OK)
      return fail(GRPO_ERR_CUDA, "grpo_debug_checks: reading the device flags failed");
  return GRPO_OK;
#else
  (void)reset;
  return fail(GRPO_ERR_UNSUPPORTED, "grpo_debug_checks: this library was built without index "
                                    "checks (build.py's checked build has them)");
#endif
}

extern "C" uint64_t grpo_kernel_launches(void) {
  return g_launches.load(std::memory_order_relaxed);
}

extern "C" grpo_status grpo_check_status(int32_t status_word) {
  clear_error();
  if (status_word == 0) return GRPO_OK;
  const uint32_t v = (uint32_t)status_word;
  const uint32_t known = GRPO_DEVFLAG_BAD_TOKEN | GRPO_DEVFLAG_NONFINITE | GRPO_DEVFLAG_TIMEOUT;
  fail(GRPO_OK, "device status 0x%x:%s%s%s%s", v,
       (v & GRPO_DEVFLAG_TIMEOUT) ? " copy wait timed out;" : "",
       (v & GRPO_DEVFLAG_BAD_TOKEN) ? " token id outside [0, V);" : "",
       (v & GRPO_DEVFLAG_NONFINITE) ? " non-finite log-sum-exp or log-prob;" : "",
       (v & ~known) ? " unknown bits;" : "");
  // a timed-out wait invalidates the launch's results; the data checks only flag rows
  return (v & GRPO_DEVFLAG_TIMEOUT) ? GRPO_ERR_TIMEOUT : GRPO_ERR_DEVICE_CHECK;
}

extern "C" grpo_status grpo_ars_init(grpo_ars_state* st, int32_t G1) {
  clear_error();
  if (st == nullptr) return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_init: state is NULL");
  if (G1 < 2) return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_init: G1 = %d, must be >= 2", G1);
  std::memset(st, 0, sizeof *st);
  st->G1 = G1;
  st->n = G1;
  return GRPO_OK;
}

// One ARS update.  The epoch buffers are kept as running sums in append order, which gives the
// same fp64 means as summing the buffered values at the epoch end.
extern "C" int32_t adaptive_rollout_count(grpo_ars_state* st, const int32_t* kept_per_prompt,
                                          int32_t P, int64_t step, int64_t total_steps,
                                          int32_t epoch_end) {
  clear_error();
  if (st == nullptr || kept_per_prompt == nullptr) {
    fail(GRPO_ERR_INVALID_ARG, "adaptive_rollout_count: NULL argument");
    return -GRPO_ERR_INVALID_ARG;
  }
  if (P < 1 || step < 1 || total_steps < step || st->G1 < 2) {
    fail(GRPO_ERR_INVALID_ARG,
         "adaptive_rollout_count: need P >= 1, 1 <= step <= total_steps, G1 >= 2 "
         "(P=%d step=%lld total=%lld G1=%d)",
         P, (long long)step, (long long)total_steps, st->G1);
    return -GRPO_ERR_INVALID_ARG;
  }
  // Eq. 10: mean and max of the retained counts over this step's prompts.
  int64_t total = 0;
  int32_t most = kept_per_prompt[0];
  for (int32_t q = 0; q < P; ++q) {
    if (kept_per_prompt[q] < 0) {
      fail(GRPO_ERR_INVALID_ARG, "adaptive_rollout_count: kept_per_prompt[%d] < 0", q);
      return -GRPO_ERR_INVALID_ARG;
    }
    total += kept_per_prompt[q];
    if (kept_per_prompt[q] > most) most = kept_per_prompt[q];
  }
  st->buf_mean_sum += (double)total / (double)P;
  st->buf_max_sum += (double)most;
  st->buf_count += 1;
  if (epoch_end) {
    const double alpha = (double)step / (double)total_steps;
    const double mean_bar = st->buf_mean_sum / (double)st->buf_count;
    const double max_bar = st->buf_max_sum / (double)st->buf_count;
    st->g_t = alpha * mean_bar + (1.0 - alpha) * max_bar;  // Eq. 11
    st->have_gt = 1;
    if (!st->have_ref) {  // Eq. 12, once, after the first epoch
      st->g_ref = (mean_bar + max_bar) / 2.0;
      st->have_ref = 1;
    }
    st->buf_mean_sum = 0.0;
    st->buf_max_sum = 0.0;
    st->buf_count = 0;
  }
  // Eqs. 13-14 for the next step.
  int32_t n = st->G1;
  if (st->have_gt && st->have_ref && st->g_t < st->g_ref) {
    const double delta = st->g_ref - st->g_t;
    double target = (double)st->G1 - delta;
    if (target > (double)st->G1) target = (double)st->G1;
    const int32_t r = (int32_t)std::nearbyint(target);  // current rounding mode: half to even
    n = r > 2 ? r : 2;
  }
  st->n = n;
  return n;
}

// ---- checkpoint / resume of the ARS state ----------------------------------------------------
// A fixed 64-byte record, little-endian whatever the host: the 8-byte tag "FRLARS01", then G1, n,
// have_ref, have_gt (4 bytes each) and g_ref, g_t, buf_mean_sum, buf_max_sum (IEEE binary64 bit
// patterns), buf_count (8 bytes each).  Written and read byte by byte, so a checkpoint moves
// between x86-64 and aarch64 hosts unchanged.

namespace {

constexpr size_t kArsRecordBytes = 64;
constexpr char kArsTag[8] = {'F', 'R', 'L', 'A', 'R', 'S', '0', '1'};

void put_u32(unsigned char* p, uint32_t v) {
  for (int i = 0; i < 4; ++i) p[i] = (unsigned char)(v >> (8 * i));
}
void put_u64(unsigned char* p, uint64_t v) {
  for (int i = 0; i < 8; ++i) p[i] = (unsigned char)(v >> (8 * i));
}
uint32_t get_u32(const unsigned char* p) {
  uint32_t v = 0;
  for (int i = 0; i < 4; ++i) v |= (uint32_t)p[i] << (8 * i);
  return v;
}
uint64_t get_u64(const unsigned char* p) {
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= (uint64_t)p[i] << (8 * i);
  return v;
}
uint64_t f64_bits(double x) {
  uint64_t b;
  std::memcpy(&b, &x, 8);
  return b;
}
double bits_f64(uint64_t b) {
  double x;
  std::memcpy(&x, &b, 8);
  return x;
}

}  // namespace

extern "C" grpo_status grpo_ars_serialize(const grpo_ars_state* st, void* buf, size_t* bytes) {
  clear_error();
  if (st == nullptr || bytes == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_serialize: NULL argument");
  if (buf == nullptr) {  // size query
    *bytes = kArsRecordBytes;
    return GRPO_OK;
  }
  if (*bytes < kArsRecordBytes)
    return fail(GRPO_ERR_WORKSPACE, "grpo_ars_serialize: buffer of %zu bytes, need %zu", *bytes,
                kArsRecordBytes);
  unsigned char* p = static_cast<unsigned char*>(buf);
  std::memcpy(p, kArsTag, 8);
  put_u32(p + 8, (uint32_t)st->G1);
  put_u32(p + 12, (uint32_t)st->n);
  put_u32(p + 16, (uint32_t)st->have_ref);
  put_u32(p + 20, (uint32_t)st->have_gt);
  put_u64(p + 24, f64_bits(st->g_ref));
  put_u64(p + 32, f64_bits(st->g_t));
  put_u64(p + 40, f64_bits(st->buf_mean_sum));
  put_u64(p + 48, f64_bits(st->buf_max_sum));
  put_u64(p + 56, (uint64_t)st->buf_count);
  *bytes = kArsRecordBytes;
  return GRPO_OK;
}

extern "C" grpo_status grpo_ars_deserialize(grpo_ars_state* st, const void* buf, size_t bytes) {
  clear_error();
  if (st == nullptr || buf == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_deserialize: NULL argument");
  if (bytes < kArsRecordBytes)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_deserialize: %zu bytes, a record has %zu", bytes,
                kArsRecordBytes);
  const unsigned char* p = static_cast<const unsigned char*>(buf);
  if (std::memcmp(p, kArsTag, 8) != 0)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_deserialize: not an ARS record (tag)");
  grpo_ars_state s;
  s.G1 = (int32_t)get_u32(p + 8);
  s.n = (int32_t)get_u32(p + 12);
  s.have_ref = (int32_t)get_u32(p + 16);
  s.have_gt = (int32_t)get_u32(p + 20);
  s.g_ref = bits_f64(get_u64(p + 24));
  s.g_t = bits_f64(get_u64(p + 32));
  s.buf_mean_sum = bits_f64(get_u64(p + 40));
  s.buf_max_sum = bits_f64(get_u64(p + 48));
  s.buf_count = (int64_t)get_u64(p + 56);
  const bool ok = s.G1 >= 2 && s.n >= 2 && s.n <= s.G1 && (s.have_ref == 0 || s.have_ref == 1) &&
                  (s.have_gt == 0 || s.have_gt == 1) && s.buf_count >= 0 &&
                  std::isfinite(s.g_ref) && std::isfinite(s.g_t) &&
                  std::isfinite(s.buf_mean_sum) && std::isfinite(s.buf_max_sum) &&
                  s.buf_mean_sum >= 0.0 && s.buf_max_sum >= 0.0;
  if (!ok) return fail(GRPO_ERR_INVALID_ARG, "grpo_ars_deserialize: inconsistent record");
  *st = s;
  return GRPO_OK;
}

extern "C" grpo_status grpo_test_fail_launch(int32_t nth) {
  clear_error();
  if (nth < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_test_fail_launch: nth = %d", nth);
  g_fail_countdown.store(nth, std::memory_order_relaxed);
  return GRPO_OK;
}
