// Greedy joint test (Section 3.4, Eq. 11; inner loop of Algorithm 1).
//
// One cooperative persistent kernel.  Every block owns fixed groups of 64
// probe rows (trajectory, selected layer, KV head, row block).  Step j:
//   phase 1  each row computes, for the candidate page E = cand[j],
//            S_E = sum e_i, U_E = sum e_i v_i (e_i = exp(s_i - m), final m
//            of the post-commit pass) and D_E = U_E - S_E o; with the sums of
//            the accepted set A it evaluates
//            r = ||D_A + D_E|| / ((l - S_A - S_E) ||o||)   (Eq. 6 on A u {E})
//            and max-reduces r into stepR[j] (Eq. 7);
//   barrier  (bounded wait: a timeout sets COMMITKV_ERR_TIMEOUT and ends);
//   phase 2  every row reads stepR[j]; if it is <= tau the row adds D_E,
//            S_E, n_E into its accepted sums.  Deletion sums over disjoint
//            pages add, which is what Eq. 11's joint deletion needs.
#include <cooperative_groups.h>

#include "ckv_internal.cuh"
#include "commitkv_testing.h"

namespace ckv {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRB = 64;
constexpr int kRowsPerWarp = kRB / kWarps;
constexpr int kTK = 64;
constexpr float kNegInf = -__builtin_huge_valf();
constexpr uint64_t kWaitNs = 1000000000ull;  // 1 s per barrier

__device__ __forceinline__ int find_group_traj(const int32_t *off, int n, int unit) {
  int t = 0;
  while (t + 1 < n && unit >= off[t + 1]) ++t;
  return t;
}

// Sense-free generation barrier over all blocks of a cooperative launch,
// with a bounded wait.  Returns false (and records a timeout) on expiry.
__device__ bool grid_barrier(WsHeader *hdr, unsigned nblocks) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    volatile uint32_t *gen = &hdr->bar_gen;
    volatile int32_t *abort_flag = &hdr->abort;
    uint32_t g = *gen;
    __threadfence();
    uint32_t arrived = atomicAdd(&hdr->bar_count, 1u);
    if (arrived == nblocks - 1) {
      atomicExch(&hdr->bar_count, 0u);
      __threadfence();
      atomicAdd(&hdr->bar_gen, 1u);
    } else {
      uint64_t t0 = globaltimer_ns();
      while (*gen == g) {
        if (*abort_flag) {
          ok = 0;
          break;
        }
        if (globaltimer_ns() - t0 > kWaitNs) {
          ok = 0;
          atomicExch(&hdr->abort, 1);
          record_error(hdr, COMMITKV_ERR_TIMEOUT, -3);
          break;
        }
        __nanosleep(64);
      }
    }
    __threadfence();
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

template <typename T, int D>
__device__ void load_group(const JointLaunch &L, const TrajDev &tr, int l, int kvh, int row0,
                           int rows, float *sQ) {
  const Batch &b = L.batch;
  const T *q = static_cast<const T *>(tr.q);
  for (int e = threadIdx.x; e < kRB * D; e += kThreads) {
    int r = e / D, c = e % D, row = row0 + r;
    float v = 0.0f;
    if (row < rows) {
      int h = kvh * b.g + row / tr.W, w = row % tr.W;
      v = to_f32(q[(((int64_t)l * b.Hq + h) * tr.W + w) * D + c]);
    }
    sQ[r * D + c] = v;
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) joint_kernel(const __grid_constant__ JointLaunch L,
                                                         WsHeader *hdr) {
  extern __shared__ float smem[];
  float *sQ = smem;
  float *sK = sQ + kRB * D;
  float *sV = sK + kTK * (D + 1);
  int *sPos = reinterpret_cast<int *>(sV + kTK * D);
  float *sP = reinterpret_cast<float *>(sPos + kTK);
  __shared__ float s_rmax;
  constexpr int J = D / 32;
  const Batch &b = L.batch;
  int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  int ngroups = L.group_off[b.n_traj];

  int steps = 0;
  for (int t = 0; t < b.n_traj; ++t) steps = max(steps, min(max(L.n_cand[t], 0), b.t[t].P));

  for (int j = 0; j < steps; ++j) {
    // ---------------- phase 1: evaluate R+(A u {E_j}) on this block's rows
    for (int grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
      int t = find_group_traj(L.group_off, b.n_traj, grp);
      const TrajDev &tr = b.t[t];
      int nc = min(max(L.n_cand[t], 0), tr.P);
      if (j >= nc) continue;
      int E = L.cand[t][j];
      if (E < 0 || E >= tr.P) {
        if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -4);
        continue;
      }
      int local = grp - L.group_off[t], nrb = L.nrb[t];
      int rb = local % nrb;
      local /= nrb;
      int kvh = local % b.H, li = local / b.H;
      int l = b.layer_ids[li];
      int rows = b.g * tr.W, row0 = rb * kRB;
      __syncthreads();
      load_group<T, D>(L, tr, l, kvh, row0, rows, sQ);
      if (threadIdx.x == 0) s_rmax = 0.0f;
      __syncthreads();

      float m2[kRowsPerWarp], lsum[kRowsPerWarp], onorm[kRowsPerWarp], o[kRowsPerWarp][J];
      float S_E[kRowsPerWarp], U[kRowsPerWarp][J];
      int nvis[kRowsPerWarp], n_E[kRowsPerWarp], qp[kRowsPerWarp];
      bool okr[kRowsPerWarp];
#pragma unroll
      for (int k = 0; k < kRowsPerWarp; ++k) {
        int row = row0 + warp * kRowsPerWarp + k;
        okr[k] = row < rows;
        int h = kvh * b.g + (okr[k] ? row / tr.W : 0), w = okr[k] ? row % tr.W : 0;
        const float *st = L.stats[t] + (((int64_t)l * b.Hq + h) * tr.W + w) * (D + 4);
        float mn = okr[k] ? st[0] : kNegInf;
        m2[k] = mn == kNegInf ? mn : mn * 1.4426950408889634f;
        lsum[k] = okr[k] ? st[1] : 0.0f;
        nvis[k] = okr[k] ? (int)st[2] : 0;
        qp[k] = okr[k] ? tr.qpos[w] : -0x7fffffff;
        float ss = 0.0f;
#pragma unroll
        for (int jj = 0; jj < J; ++jj) {
          o[k][jj] = okr[k] ? st[4 + lane + 32 * jj] : 0.0f;
          ss = fmaf(o[k][jj], o[k][jj], ss);
          U[k][jj] = 0.0f;
        }
        onorm[k] = sqrtf(warp_sum(ss));
        S_E[k] = 0.0f;
        n_E[k] = 0;
      }
      int ps = tr.ps[E], pl = tr.pl[E];
      if (pl < 0 || ps < 0 || ps > tr.S - pl) {
        if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, E);
        pl = 0;
        ps = 0;
      }
      const T *kp = static_cast<const T *>(tr.k) + (int64_t)l * tr.sl + (int64_t)kvh * tr.sh;
      const T *vp = static_cast<const T *>(tr.v) + (int64_t)l * tr.sl + (int64_t)kvh * tr.sh;
      for (int tok0 = ps; tok0 < ps + pl; tok0 += kTK) {
        int nt = min(kTK, ps + pl - tok0);
        __syncthreads();
        for (int e = threadIdx.x; e < kTK * D; e += kThreads) {
          int i = e / D, c = e % D;
          float kv = 0.0f, vv = 0.0f;
          if (i < nt) {
            int64_t off = (int64_t)(tok0 + i) * tr.st + c;
            kv = to_f32(kp[off]);
            vv = to_f32(vp[off]);
          }
          sK[i * (D + 1) + c] = kv;
          sV[i * D + c] = vv;
        }
        for (int i = threadIdx.x; i < kTK; i += kThreads) sPos[i] = i < nt ? tr.pos[tok0 + i] : 0;
        __syncthreads();
#pragma unroll 1
        for (int k = 0; k < kRowsPerWarp; ++k) {
          if (!okr[k]) continue;
          const float *q = sQ + (warp * kRowsPerWarp + k) * D;
          bool v0 = lane < nt && sPos[lane] <= qp[k], v1 = lane + 32 < nt && sPos[lane + 32] <= qp[k];
          float s0 = 0.0f, s1 = 0.0f;
          if (v0)
            for (int c = 0; c < D; ++c) s0 = fmaf(q[c], sK[lane * (D + 1) + c], s0);
          if (v1)
            for (int c = 0; c < D; ++c) s1 = fmaf(q[c], sK[(lane + 32) * (D + 1) + c], s1);
          float e0 = v0 ? exp2f(s0 * b.scale_log2 - m2[k]) : 0.0f;
          float e1 = v1 ? exp2f(s1 * b.scale_log2 - m2[k]) : 0.0f;
          S_E[k] += warp_sum(e0 + e1);
          n_E[k] += __popc(__ballot_sync(0xffffffffu, v0)) + __popc(__ballot_sync(0xffffffffu, v1));
          float *pw = sP + warp * kTK;
          pw[lane] = e0;
          pw[lane + 32] = e1;
          __syncwarp();
          for (int i = 0; i < nt; ++i) {
            float p = pw[i];
#pragma unroll
            for (int jj = 0; jj < J; ++jj) U[k][jj] = fmaf(p, sV[i * D + lane + 32 * jj], U[k][jj]);
          }
          __syncwarp();
        }
      }
      float rmax = 0.0f;
#pragma unroll
      for (int k = 0; k < kRowsPerWarp; ++k) {
        if (!okr[k]) continue;
        int64_t grow = L.row_off[t] + (int64_t)(li * b.H + kvh) * rows + row0 + warp * kRowsPerWarp + k;
        float *DA = L.DA + grow * D;
        float *DE = L.DE + grow * D;
        float *SA = L.SA + grow * 4;
        float ss = 0.0f;
#pragma unroll
        for (int jj = 0; jj < J; ++jj) {
          float de = fmaf(-S_E[k], o[k][jj], U[k][jj]);
          DE[lane + 32 * jj] = de;
          float dsum = DA[lane + 32 * jj] + de;
          ss = fmaf(dsum, dsum, ss);
        }
        float num2 = warp_sum(ss);
        float S_tot = SA[0] + S_E[k];
        int n_tot = (int)SA[1] + n_E[k];
        float r = effect_value(n_tot, nvis[k], S_tot, lsum[k], num2, onorm[k]);
        rmax = fmaxf(rmax, r);
        if (lane == 0) {
          SA[2] = S_E[k];
          SA[3] = (float)n_E[k];
        }
      }
      if (lane == 0) atomicMax(reinterpret_cast<int *>(&s_rmax), __float_as_int(rmax));
      __syncthreads();
      if (threadIdx.x == 0) atomic_max_nonneg(L.stepR[t] + j, s_rmax);
    }
    // ---------------- barrier: every block's contribution to stepR[j] is in
    if (!grid_barrier(hdr, gridDim.x)) return;
    // ---------------- phase 2: accept or reject, add the accepted sums
    for (int grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
      int t = find_group_traj(L.group_off, b.n_traj, grp);
      const TrajDev &tr = b.t[t];
      int nc = min(max(L.n_cand[t], 0), tr.P);
      if (j >= nc) continue;
      int E = L.cand[t][j];
      if (E < 0 || E >= tr.P) continue;
      float R = *(volatile float *)(L.stepR[t] + j);
      if (!(R <= L.tau)) continue;
      int local = grp - L.group_off[t], nrb = L.nrb[t];
      int rb = local % nrb;
      local /= nrb;
      int kvh = local % b.H, li = local / b.H;
      int rows = b.g * tr.W, row0 = rb * kRB;
#pragma unroll 1
      for (int k = 0; k < kRowsPerWarp; ++k) {
        int row = row0 + warp * kRowsPerWarp + k;
        if (row >= rows) continue;
        int64_t grow = L.row_off[t] + (int64_t)(li * b.H + kvh) * rows + row;
        float *DA = L.DA + grow * D;
        const float *DE = L.DE + grow * D;
        float *SA = L.SA + grow * 4;
#pragma unroll
        for (int jj = 0; jj < J; ++jj) DA[lane + 32 * jj] += DE[lane + 32 * jj];
        if (lane == 0) {
          SA[0] += SA[2];
          SA[1] += SA[3];
        }
      }
    }
    if (blockIdx.x == 0) {
      for (int t = threadIdx.x; t < b.n_traj; t += kThreads) {
        const TrajDev &tr = b.t[t];
        int nc = min(max(L.n_cand[t], 0), tr.P);
        if (j >= nc) continue;
        int E = L.cand[t][j];
        float R = *(volatile float *)(L.stepR[t] + j);
        if (L.stepR_out[t]) L.stepR_out[t][j] = R;
        if (E >= 0 && E < tr.P && R <= L.tau) L.accepted[t][E] = 1;
      }
    }
  }
}

template <typename T, int D>
cudaError_t launch_joint_typed(const JointLaunch &L, WsHeader *hdr, cudaStream_t s, int sm_count) {
  size_t smem = (size_t)(kRB * D + kTK * (D + 1) + kTK * D) * 4 + kTK * 4 + kWarps * kTK * 4;
  cudaError_t e = cudaFuncSetAttribute(joint_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, joint_kernel<T, D>, kThreads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  int ngroups = L.group_off[L.batch.n_traj];
  int grid = per_sm * sm_count;
  if (grid > ngroups) grid = ngroups;
  if (grid < 1) return cudaSuccess;
  void *args[] = {(void *)&L, (void *)&hdr};
  return cudaLaunchCooperativeKernel((const void *)joint_kernel<T, D>, dim3(grid), dim3(kThreads),
                                     args, smem, s);
}

}  // namespace

cudaError_t launch_joint(const JointLaunch &L, WsHeader *hdr, cudaStream_t stream, int sm_count) {
  bool bf = L.batch.dtype == COMMITKV_BF16;
  if (L.batch.d == 128)
    return bf ? launch_joint_typed<__nv_bfloat16, 128>(L, hdr, stream, sm_count)
              : launch_joint_typed<float, 128>(L, hdr, stream, sm_count);
  return bf ? launch_joint_typed<__nv_bfloat16, 64>(L, hdr, stream, sm_count)
            : launch_joint_typed<float, 64>(L, hdr, stream, sm_count);
}

int joint_rows_per_group() { return kRB; }

namespace {
__global__ void barrier_timeout_kernel(WsHeader *hdr, unsigned expected) { grid_barrier(hdr, expected); }
}  // namespace

}  // namespace ckv

extern "C" commitkv_status commitkv_test_barrier_timeout(void *workspace, size_t workspace_bytes,
                                                         int32_t blocks, cudaStream_t stream) {
  if (!workspace || workspace_bytes < sizeof(ckv::WsHeader) || blocks < 1 || blocks > 64)
    return COMMITKV_ERR_INVALID_ARG;
  ckv::WsHeader *hdr = static_cast<ckv::WsHeader *>(workspace);
  if (cudaMemsetAsync(&hdr->abort, 0, 3 * sizeof(int32_t), stream) != cudaSuccess) return COMMITKV_ERR_CUDA;
  unsigned expected = (unsigned)blocks + 1;
  void *args[] = {(void *)&hdr, (void *)&expected};
  cudaError_t e = cudaLaunchCooperativeKernel((const void *)ckv::barrier_timeout_kernel, dim3(blocks),
                                              dim3(32), args, 0, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return COMMITKV_ERR_CUDA;
  }
  return COMMITKV_OK;
}
