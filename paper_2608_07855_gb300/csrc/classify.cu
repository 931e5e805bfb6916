// Lifecycle classification (Section 3.3, Eq. 9-10) and candidate ordering
// (Section 3.4).  One block per trajectory; page counts are in the
// thousands, so the percentile ranks are plain counting compares.
#include "ckv_internal.cuh"

namespace ckv {
namespace {

constexpr int kThreads = 1024;

__device__ __forceinline__ bool key_less(const float *Rm, const float *Rp, int a, int b) {
  // increasing R+, then decreasing R-, then increasing page index
  if (Rp[a] != Rp[b]) return Rp[a] < Rp[b];
  if (Rm[a] != Rm[b]) return Rm[a] > Rm[b];
  return a < b;
}

__global__ void __launch_bounds__(kThreads) classify_kernel(const __grid_constant__ ClassifyLaunch L,
                                                            WsHeader *hdr) {
  int t = blockIdx.x;
  int P = L.P[t];
  const float *Rm = L.Rm[t];
  const float *Rp = L.Rp[t];
  const uint8_t *el = L.el[t];
  __shared__ int s_n, s_c, s_bad;
  if (threadIdx.x == 0) {
    s_n = 0;
    s_c = 0;
    s_bad = 0;
  }
  __syncthreads();
  int n_local = 0;
  for (int E = threadIdx.x; E < P; E += kThreads) {
    if (!el[E]) continue;
    ++n_local;
    if (isnan(Rm[E]) || isnan(Rp[E])) s_bad = 1;
  }
  atomicAdd(&s_n, n_local);
  __syncthreads();
  if (s_bad) {
    if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -2);
    for (int E = threadIdx.x; E < P; E += kThreads) L.state[t][E] = 0;
    if (threadIdx.x == 0) L.n_cand[t] = 0;
    return;
  }
  int n = s_n;
  for (int E = threadIdx.x; E < P; E += kThreads) {
    if (!el[E]) {
      L.state[t][E] = 0;
      continue;
    }
    float rm = Rm[E], rp = Rp[E];
    int km = 0, kp = 0;
    for (int F = 0; F < P; ++F) {
      if (!el[F]) continue;
      km += Rm[F] < rm;
      kp += Rp[F] < rp;
    }
    double Pm = (double)km / (double)n, Pp = (double)kp / (double)n;
    // without percentile calibration the states use the absolute thresholds only
    const bool pct = !(L.variant & COMMITKV_CLASSIFY_NO_PERCENTILE);
    bool Hm = rm >= L.tau_use && (!pct || Pm >= L.rho_use);
    bool Lm = rm <= L.tau_dead && (!pct || Pm <= L.rho_dead);
    bool Hp = rp >= L.tau_use && (!pct || Pp >= L.rho_use);
    bool Lp = rp <= L.tau_dead && (!pct || Pp <= L.rho_dead);
    uint8_t st = 5;  // uncertain
    if (Hm && Lp) st = 1;       // completion candidate
    else if (Lm && Lp) st = 2;  // dormant
    else if (Lm && Hp) st = 3;  // newly active
    else if (Hm && Hp) st = 4;  // still active
    L.state[t][E] = st;
    // without the pre-commit state every page low after the commit is a candidate
    const bool cand = (L.variant & COMMITKV_CLASSIFY_NO_PRECOMMIT) ? Lp : st == 1;
    if (cand) L.scratch[t][atomicAdd(&s_c, 1)] = E;
  }
  __syncthreads();
  int C = s_c;
  for (int i = threadIdx.x; i < C; i += kThreads) {
    int E = L.scratch[t][i];
    int rank = 0;
    for (int j = 0; j < C; ++j) rank += key_less(Rm, Rp, L.scratch[t][j], E);
    L.cand[t][rank] = E;
  }
  if (threadIdx.x == 0) L.n_cand[t] = C;
}

}  // namespace

cudaError_t launch_classify(const ClassifyLaunch &L, WsHeader *hdr, cudaStream_t stream) {
  if (L.n_traj <= 0) return cudaSuccess;
  classify_kernel<<<L.n_traj, kThreads, 0, stream>>>(L, hdr);
  return cudaGetLastError();
}

}  // namespace ckv
