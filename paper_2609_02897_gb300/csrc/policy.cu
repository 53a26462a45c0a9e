// Dynamic tree-shape policy (Sec. 3.3, Eq. 2): per request, the running
// acceptance rate (RAR, an EMA of the accepted fraction of drafted nodes), the
// Draft Confidence Score DCS = min(1, p_draft(top1) * RAR / d), its linear
// mapping onto the (n_steps, topk, ndt) range, and the circuit breaker that
// returns a request to its starting state after `breaker` consecutive
// zero-accept steps.
//
// One thread per request; the kernels read the verify step's outputs
// (path_len) and the draft LM head's row statistics (row_max, row_lse) where
// they already are, in device memory, so a decode loop can keep the policy
// on the GPU and inside a CUDA graph.  All arithmetic is binary64 with every
// product, quotient and sum rounded on its own (__dmul_rn, __ddiv_rn,
// __dadd_rn: no contraction into fused multiply-adds), so the device results
// and the host enumeration of reachable triplets agree bit for bit.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include "common.cuh"

namespace asd {
namespace {

constexpr int kPolicyThreads = 128;
constexpr int kPolicyMaxCoord = 128;

struct PolicyConst {
  double alpha, divisor, rar_init;
  int shallow[3], deep[3];
  int breaker;
};

bool params_ok(const asd_policy_params* p) {
  if (!p) return false;
  if (!(p->alpha > 0.0 && p->alpha <= 1.0)) return false;
  if (!(p->divisor > 0.0) || !std::isfinite(p->divisor)) return false;
  if (!(p->rar_init >= 0.0 && p->rar_init <= 1.0)) return false;
  for (int k = 0; k < 3; ++k) {
    if (p->shallow[k] < 1 || p->shallow[k] > kPolicyMaxCoord) return false;
    if (p->deep[k] < 1 || p->deep[k] > kPolicyMaxCoord) return false;
  }
  return p->breaker >= 1 && p->reserved == 0;
}

PolicyConst to_const(const asd_policy_params* p) {
  PolicyConst c;
  c.alpha = p->alpha;
  c.divisor = p->divisor;
  c.rar_init = p->rar_init;
  for (int k = 0; k < 3; ++k) {
    c.shallow[k] = p->shallow[k];
    c.deep[k] = p->deep[k];
  }
  c.breaker = p->breaker;
  return c;
}

// start + round(span * u), halves upward.  y - floor(y) is exact, so the
// rounding decision is exact given the rounded product.
__device__ __forceinline__ int interp_dev(int start, int end, double u) {
  const double y = __dmul_rn(static_cast<double>(end - start), u);
  const double f = floor(y);
  return start + static_cast<int>(f) + (__dsub_rn(y, f) >= 0.5 ? 1 : 0);
}

__global__ void policy_init_kernel(PolicyConst c, asd_policy_state* st, int batch) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  st[b].rar = c.rar_init;
  st[b].zero_streak = 0;
  st[b].breaks = 0;
}

__global__ void policy_update_kernel(PolicyConst c, const int* __restrict__ cu_nodes,
                                     const int* __restrict__ path_len, asd_policy_state* st,
                                     int batch) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const int n = cu_nodes[b + 1] - cu_nodes[b];
  const int len = path_len[b];
  if (n <= 1 || len <= 0 || len > n) return;
  const int accepted = len - 1;
  const double frac = __ddiv_rn(static_cast<double>(accepted), static_cast<double>(n - 1));
  asd_policy_state s = st[b];
  s.rar = __dadd_rn(__dmul_rn(c.alpha, frac), __dmul_rn(__dsub_rn(1.0, c.alpha), s.rar));
  s.zero_streak = accepted == 0 ? s.zero_streak + 1 : 0;
  if (s.zero_streak >= c.breaker) {
    s.rar = c.rar_init;
    s.zero_streak = 0;
    s.breaks += 1;
  }
  st[b] = s;
}

__global__ void policy_select_kernel(PolicyConst c, const float* __restrict__ row_max,
                                     const float* __restrict__ row_lse,
                                     const int* __restrict__ rows, int num_rows,
                                     const asd_policy_state* __restrict__ st, int batch,
                                     int* __restrict__ triplet, double* __restrict__ dcs) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const int r = rows ? rows[b] : b;
  if (r < 0 || r >= num_rows) {
    triplet[3 * b] = triplet[3 * b + 1] = triplet[3 * b + 2] = 0;
    if (dcs) dcs[b] = __longlong_as_double(0x7ff8000000000000LL);
    return;
  }
  // p_draft(top1) = exp(m - lse): the softmax's top-1 probability
  double p = exp(__dsub_rn(static_cast<double>(row_max[r]), static_cast<double>(row_lse[r])));
  if (!(p >= 0.0)) p = 0.0;
  double score = __ddiv_rn(__dmul_rn(p, st[b].rar), c.divisor);
  score = score < 1.0 ? score : 1.0;
  const double rest = __dsub_rn(1.0, score);
  triplet[3 * b] = interp_dev(c.shallow[0], c.deep[0], score);
  triplet[3 * b + 1] = interp_dev(c.deep[1], c.shallow[1], rest);
  triplet[3 * b + 2] = interp_dev(c.shallow[2], c.deep[2], score);
  if (dcs) dcs[b] = score;
}

// ------------------------------------------------------------ host mapping

// The device mapping evaluated on the host; `volatile` keeps each product
// and difference rounded on its own whatever the host compiler contracts.
int interp_host(int start, int end, double u) {
  volatile double y = static_cast<double>(end - start) * u;
  const double yv = y;
  const double f = std::floor(yv);
  volatile double frac = yv - f;
  return start + static_cast<int>(f) + (frac >= 0.5 ? 1 : 0);
}

void triplet_host(const asd_policy_params& p, double s, int t[3]) {
  volatile double rest = 1.0 - s;
  t[0] = interp_host(p.shallow[0], p.deep[0], s);
  t[1] = interp_host(p.deep[1], p.shallow[1], rest);
  t[2] = interp_host(p.shallow[2], p.deep[2], s);
}

double from_bits(uint64_t b) {
  double d;
  std::memcpy(&d, &b, sizeof d);
  return d;
}

uint64_t to_bits(double d) {
  uint64_t b;
  std::memcpy(&b, &d, sizeof b);
  return b;
}

}  // namespace
}  // namespace asd

using namespace asd;

extern "C" {

int32_t asd_policy_triplets(const asd_policy_params* params, int32_t* out, int32_t cap) {
  if (!params_ok(params) || cap < 0 || (cap > 0 && !out)) return -ASD_ERR_INVALID_ARG;
  const asd_policy_params& p = *params;
  // Each coordinate is a monotone step function of the score (rounded
  // monotone operations); the non-negative doubles are ordered like their
  // bit patterns, so each of its value changes is located by bisection over
  // [bits(0), bits(1)].  Between consecutive change points the triplet is
  // constant.
  const uint64_t lo = to_bits(0.0), hi = to_bits(1.0);
  std::vector<uint64_t> cand = {lo, hi};
  for (int k = 0; k < 3; ++k) {
    auto coord = [&](uint64_t b) {
      int t[3];
      triplet_host(p, from_bits(b), t);
      return t[k];
    };
    const int g0 = coord(lo), g1 = coord(hi);
    const int step = g1 > g0 ? 1 : -1;
    for (int v = g0; v != g1; v += step) {
      uint64_t a = lo, b = hi;  // coord(a) has not moved past v, coord(b) has
      while (b - a > 1) {
        const uint64_t m = a + (b - a) / 2;
        if ((coord(m) - v) * step > 0)
          b = m;
        else
          a = m;
      }
      cand.push_back(a);
      cand.push_back(b);
    }
  }
  std::sort(cand.begin(), cand.end());
  int32_t count = 0;
  int prev[3] = {-1, -1, -1};
  for (uint64_t b : cand) {
    int t[3];
    triplet_host(p, from_bits(b), t);
    if (t[0] == prev[0] && t[1] == prev[1] && t[2] == prev[2]) continue;
    if (count < cap)
      for (int k = 0; k < 3; ++k) out[3 * count + k] = t[k];
    for (int k = 0; k < 3; ++k) prev[k] = t[k];
    ++count;
  }
  return count;
}

asd_status asd_policy_init(const asd_policy_params* params, asd_policy_state* state,
                           int32_t batch, void* stream) {
  if (!params_ok(params) || !state || batch < 0) return ASD_ERR_INVALID_ARG;
  if (batch == 0) return ASD_OK;
  policy_init_kernel<<<(batch + kPolicyThreads - 1) / kPolicyThreads, kPolicyThreads, 0,
                       static_cast<cudaStream_t>(stream)>>>(to_const(params), state, batch);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

asd_status asd_policy_update(const asd_policy_params* params, const int32_t* cu_nodes,
                             const int32_t* path_len, int32_t batch, asd_policy_state* state,
                             void* stream) {
  if (!params_ok(params) || !cu_nodes || !path_len || !state || batch < 0)
    return ASD_ERR_INVALID_ARG;
  if (batch == 0) return ASD_OK;
  policy_update_kernel<<<(batch + kPolicyThreads - 1) / kPolicyThreads, kPolicyThreads, 0,
                         static_cast<cudaStream_t>(stream)>>>(to_const(params), cu_nodes,
                                                              path_len, state, batch);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

asd_status asd_policy_select(const asd_policy_params* params, const float* row_max,
                             const float* row_lse, const int32_t* rows, int32_t num_rows,
                             int32_t batch, const asd_policy_state* state, int32_t* triplet,
                             double* dcs, void* stream) {
  if (!params_ok(params) || !row_max || !row_lse || !state || !triplet || batch < 0 ||
      num_rows < 0)
    return ASD_ERR_INVALID_ARG;
  if (batch == 0) return ASD_OK;
  policy_select_kernel<<<(batch + kPolicyThreads - 1) / kPolicyThreads, kPolicyThreads, 0,
                         static_cast<cudaStream_t>(stream)>>>(
      to_const(params), row_max, row_lse, rows, num_rows, state, batch, triplet, dcs);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

}  // extern "C"
