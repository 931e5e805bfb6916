// Lifecycle classification (Section 3.2, Eq. 9-10) and candidate ordering
// (Section 3.3), in two kernels:
//   state  one warp per page (32 pages per block, every trajectory): the
//          percentile ranks of R- and R+ among the eligible pages are plain
//          counting compares split over the lanes; the page's state and
//          whether it is a candidate;
//   order  one block per trajectory: the candidates sorted by increasing
//          R+, then decreasing R-, then page index.
// Both count the eligible pages and look for NaN effects themselves; with a
// NaN every state is 0 and there are no candidates.
#include "ckv_internal.cuh"

namespace ckv {
namespace {

constexpr int kThreads = 1024;
constexpr int kPagesPerBlock = kThreads / 32;
constexpr int kMaxList = 4096;  // candidates ordered from shared memory

__device__ __forceinline__ bool key_less(const float *Rm, const float *Rp, int a, int b) {
  // increasing R+, then decreasing R-, then increasing page index
  if (Rp[a] != Rp[b]) return Rp[a] < Rp[b];
  if (Rm[a] != Rm[b]) return Rm[a] > Rm[b];
  return a < b;
}

// Eligible pages of trajectory t and whether any of them has a NaN effect.
__device__ void count_eligible(const ClassifyLaunch &L, int t, int *s_n, int *s_bad) {
  const int P = L.P[t];
  if (threadIdx.x == 0) {
    *s_n = 0;
    *s_bad = 0;
  }
  __syncthreads();
  int n_local = 0;
  for (int E = threadIdx.x; E < P; E += kThreads) {
    if (!L.el[t][E]) continue;
    ++n_local;
    if (isnan(L.Rm[t][E]) || isnan(L.Rp[t][E])) *s_bad = 1;
  }
  atomicAdd(s_n, n_local);
  __syncthreads();
}

__global__ void __launch_bounds__(kThreads) classify_state_kernel(const __grid_constant__ ClassifyLaunch L,
                                                                  WsHeader *hdr) {
  const int t = blockIdx.y, P = L.P[t];
  if ((int)blockIdx.x * kPagesPerBlock >= P) return;
  __shared__ int s_n, s_bad;
  count_eligible(L, t, &s_n, &s_bad);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int E = blockIdx.x * kPagesPerBlock + warp;
  if (E >= P) return;
  const float *Rm = L.Rm[t];
  const float *Rp = L.Rp[t];
  const uint8_t *el = L.el[t];
  if (s_bad) {
    if (E == 0 && lane == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -2);
    if (lane == 0) {
      L.state[t][E] = 0;
      L.scratch[t][E] = 0;
    }
    return;
  }
  if (!el[E]) {
    if (lane == 0) {
      L.state[t][E] = 0;
      L.scratch[t][E] = 0;
    }
    return;
  }
  const float rm = Rm[E], rp = Rp[E];
  int km = 0, kp = 0;
  for (int F = lane; F < P; F += 32) {
    if (!el[F]) continue;
    km += Rm[F] < rm;
    kp += Rp[F] < rp;
  }
  km = warp_sum_i(km);
  kp = warp_sum_i(kp);
  if (lane == 0) {
    const int n = s_n;
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
    L.scratch[t][E] = cand ? 1 : 0;
  }
}

__global__ void __launch_bounds__(kThreads) classify_order_kernel(const __grid_constant__ ClassifyLaunch L) {
  const int t = blockIdx.x, P = L.P[t];
  const float *Rm = L.Rm[t];
  const float *Rp = L.Rp[t];
  const int32_t *flag = L.scratch[t];
  __shared__ int s_n, s_bad, s_c;
  __shared__ int s_list[kMaxList];
  count_eligible(L, t, &s_n, &s_bad);
  if (s_bad) {
    if (threadIdx.x == 0) L.n_cand[t] = 0;
    return;
  }
  if (threadIdx.x == 0) s_c = 0;
  __syncthreads();
  for (int E = threadIdx.x; E < P; E += kThreads) {
    if (!flag[E]) continue;
    const int k = atomicAdd(&s_c, 1);
    if (k < kMaxList) s_list[k] = E;
  }
  __syncthreads();
  const int C = s_c;
  if (C <= kMaxList) {
    for (int i = threadIdx.x; i < C; i += kThreads) {
      const int E = s_list[i];
      int rank = 0;
      for (int j = 0; j < C; ++j) rank += key_less(Rm, Rp, s_list[j], E);
      L.cand[t][rank] = E;
    }
  } else {
    for (int E = threadIdx.x; E < P; E += kThreads) {
      if (!flag[E]) continue;
      int rank = 0;
      for (int F = 0; F < P; ++F) rank += flag[F] && key_less(Rm, Rp, F, E);
      L.cand[t][rank] = E;
    }
  }
  if (threadIdx.x == 0) L.n_cand[t] = C;
}

}  // namespace

cudaError_t launch_classify(const ClassifyLaunch &L, WsHeader *hdr, cudaStream_t stream) {
  if (L.n_traj <= 0) return cudaSuccess;
  int pmax = 0;
  for (int t = 0; t < L.n_traj; ++t) pmax = L.P[t] > pmax ? L.P[t] : pmax;
  if (pmax > 0) {
    dim3 grid((pmax + kPagesPerBlock - 1) / kPagesPerBlock, L.n_traj);
    classify_state_kernel<<<grid, kThreads, 0, stream>>>(L, hdr);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  classify_order_kernel<<<L.n_traj, kThreads, 0, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace ckv
