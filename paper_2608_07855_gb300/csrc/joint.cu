// Greedy joint test (Section 3.3, Eq. 11; inner loop of Algorithm 1) on the
// CUDA cores: the path for fp32 caches, head_dim 64 and rows that the
// tensor-core kernel (joint_tc.cu) cannot stage; launch_joint chooses.
//
// One cooperative persistent kernel.  Every block owns fixed groups of 16
// probe rows (trajectory, selected layer, KV head, row block).  The
// candidates are taken in rounds of kRound:
//   phase 1  each row loads its accepted-set sums (D_A = sum over A of
//            U_E - S_E o, S_A, n_A) once, then computes for every candidate E
//            of the round S_E = sum e_i, n_E and D_E = U_E - S_E o (e_i =
//            exp(s_i - m) with the final m of the post-commit pass).  For each
//            candidate c and each subset B of the round's earlier candidates
//            it evaluates Eq. 6 on A u B u {E_c},
//              r = ||D_A + D_B + D_c|| / ((l - S_A - S_B - S_c) ||o||),
//            adding the sums in candidate order, which is the order in which
//            the one-candidate-at-a-time scan would have added them; the max
//            over rows of each (c, B) goes to a per-round table (Eq. 7);
//   barrier  (bounded wait: a timeout sets COMMITKV_ERR_TIMEOUT and ends);
//   phase 2  every block replays the round's decisions from the table:
//            candidate c is accepted iff its value for B = the round's
//            candidates accepted before it is <= tau, then adds the accepted
//            D_c, S_c, n_c into its rows' sums, in candidate order.
// The decisions and step values are those of the scan that takes one
// candidate per barrier; deletion sums over disjoint pages add, which is what
// Eq. 11's joint deletion needs.
#include "joint_common.cuh"
#include "commitkv_testing.h"

namespace ckv {
namespace {

using joint::combo;
using joint::kCombos;
using joint::kRound;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerWarp = 2;
constexpr int kRB = kWarps * kRowsPerWarp;  // rows per group
constexpr int kTK = 64;                     // page tokens per shared-memory chunk
constexpr float kNegInf = -__builtin_huge_valf();

// J consecutive floats (J = 2 or 4) as one vector access.
template <int J>
__device__ __forceinline__ void lds_vec(const float *p, float (&v)[J]) {
  if constexpr (J == 4) {
    float4 x = *reinterpret_cast<const float4 *>(p);
    v[0] = x.x, v[1] = x.y, v[2] = x.z, v[3] = x.w;
  } else {
    float2 x = *reinterpret_cast<const float2 *>(p);
    v[0] = x.x, v[1] = x.y;
  }
}
template <int J>
__device__ __forceinline__ void sts_vec(float *p, const float (&v)[J]) {
  if constexpr (J == 4) *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
  else *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
}
// 16 bytes of K or V (8 bf16 or 4 floats) as floats: one vector load when the
// address allows it, else element loads.
template <typename T>
__device__ __forceinline__ void load16_f32(const T *p, float (&out)[16 / sizeof(T)]) {
  constexpr int n = 16 / sizeof(T);
  if ((reinterpret_cast<uintptr_t>(p) & 15) == 0) {
    const uint4 raw = *reinterpret_cast<const uint4 *>(p);
    const T *e = reinterpret_cast<const T *>(&raw);
#pragma unroll
    for (int u = 0; u < n; ++u) out[u] = to_f32(e[u]);
  } else {
#pragma unroll
    for (int u = 0; u < n; ++u) out[u] = to_f32(p[u]);
  }
}

struct Group {
  int t, l, li, kvh, rows, row0;
};

__device__ __forceinline__ Group decode_group(const JointLaunch &L, int grp) {
  const Batch &b = L.batch;
  Group G;
  G.t = joint::find_group_traj(L.group_off, b.n_traj, grp);
  int local = grp - L.group_off[G.t], nrb = L.nrb[G.t];
  int rb = local % nrb;
  local /= nrb;
  G.kvh = local % b.H;
  G.li = local / b.H;
  G.l = b.layer_ids[G.li];
  G.rows = b.g * b.t[G.t].W;
  G.row0 = rb * kRB;
  return G;
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 2) joint_kernel(const __grid_constant__ JointLaunch L,
                                                         WsHeader *hdr) {
  extern __shared__ float smem[];
  float *sQ = smem;                           // [kRB][D]
  float *sK = sQ + kRB * D;                   // [kTK][D + 4]
  float *sV = sK + kTK * (D + 4);             // [kTK][D]
  int *sPos = reinterpret_cast<int *>(sV + kTK * D);
  float *sP = reinterpret_cast<float *>(sPos + kTK);  // [kWarps][kTK][kRowsPerWarp]
  __shared__ float s_rmax[kCombos];
  // Each lane owns J = D / 32 consecutive channels (J * lane ..) of every
  // row, so that V, D_c and D_A move as one vector per lane.
  constexpr int J = D / 32;
  const Batch &b = L.batch;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int ngroups = L.group_off[b.n_traj];
  const int64_t rows_full = L.rows_full;

  const int rounds = joint::round_total(L);

  for (int r = 0; r < rounds; ++r) {
    float *tab_r = joint::round_table(L, r);
    // ---------------- phase 1: the round's candidates on this block's rows
    for (int grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
      const Group G = decode_group(L, grp);
      const TrajDev &tr = b.t[G.t];
      const int kc = joint::round_count(L, G.t, r);
      if (kc == 0) continue;
      __syncthreads();
      for (int e = threadIdx.x; e < kRB * D; e += kThreads) {
        int rr = e / D, c = e % D, row = G.row0 + rr;
        float v = 0.0f;
        if (row < G.rows) {
          int h = G.kvh * b.g + row / tr.W, w = row % tr.W;
          v = to_f32(static_cast<const T *>(tr.q)[(((int64_t)G.l * b.Hq + h) * tr.W + w) * D + c]);
        }
        sQ[rr * D + c] = v;
      }
      if (threadIdx.x < kCombos) s_rmax[threadIdx.x] = 0.0f;
      __syncthreads();

      float m2[kRowsPerWarp], lsum[kRowsPerWarp], onorm[kRowsPerWarp], o[kRowsPerWarp][J], DA[kRowsPerWarp][J];
      float SA[kRowsPerWarp];
      int nA[kRowsPerWarp], nvis[kRowsPerWarp], qp[kRowsPerWarp];
      bool okr[kRowsPerWarp];
      int64_t grow[kRowsPerWarp];
#pragma unroll
      for (int k = 0; k < kRowsPerWarp; ++k) {
        int row = G.row0 + warp * kRowsPerWarp + k;
        okr[k] = row < G.rows;
        int h = G.kvh * b.g + (okr[k] ? row / tr.W : 0), w = okr[k] ? row % tr.W : 0;
        grow[k] = L.row_off[G.t] + (int64_t)(G.li * b.H + G.kvh) * G.rows + (okr[k] ? row : 0);
        const float *st = L.stats[G.t] + (((int64_t)G.l * b.Hq + h) * tr.W + w) * (D + 4);
        float mn = okr[k] ? st[0] : kNegInf;
        m2[k] = mn == kNegInf ? mn : mn * 1.4426950408889634f;
        lsum[k] = okr[k] ? st[1] : 0.0f;
        nvis[k] = okr[k] ? (int)st[2] : 0;
        qp[k] = okr[k] ? tr.qpos[w] : -0x7fffffff;
        const float *da = L.DA + grow[k] * D;
        float ss = 0.0f;
#pragma unroll
        for (int jj = 0; jj < J; ++jj) {
          const int ch = J * lane + jj;
          o[k][jj] = okr[k] ? st[4 + ch] : 0.0f;
          ss = fmaf(o[k][jj], o[k][jj], ss);
          DA[k][jj] = okr[k] ? da[ch] : 0.0f;
        }
        onorm[k] = sqrtf(warp_sum(ss));
        SA[k] = okr[k] ? L.SA[grow[k] * 2] : 0.0f;
        nA[k] = okr[k] ? (int)L.SA[grow[k] * 2 + 1] : 0;
      }

      // D_c, S_c, n_c of each candidate of the round
      float DE[kRound][kRowsPerWarp][J], SE[kRound][kRowsPerWarp];
      int nE[kRound][kRowsPerWarp];
#pragma unroll
      for (int c = 0; c < kRound; ++c) {
        float U[kRowsPerWarp][J], S_c[kRowsPerWarp];
        int n_c[kRowsPerWarp];
#pragma unroll
        for (int k = 0; k < kRowsPerWarp; ++k) {
          S_c[k] = 0.0f;
          n_c[k] = 0;
#pragma unroll
          for (int jj = 0; jj < J; ++jj) U[k][jj] = 0.0f;
        }
        int ps = 0, pl = 0;
        if (c < kc) {
          int E = L.cand[G.t][r * kRound + c];
          if (E < 0 || E >= tr.P) {
            if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -4);
          } else {
            ps = tr.ps[E];
            pl = tr.pl[E];
            if (pl < 0 || ps < 0 || ps > tr.S - pl) {
              if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, E);
              pl = 0;
              ps = 0;
            }
          }
        }
        const T *kp = static_cast<const T *>(tr.k) + (int64_t)G.l * tr.sl + (int64_t)G.kvh * tr.sh;
        const T *vp = static_cast<const T *>(tr.v) + (int64_t)G.l * tr.sl + (int64_t)G.kvh * tr.sh;
        for (int tok0 = ps; tok0 < ps + pl; tok0 += kTK) {
          const int nt = min(kTK, ps + pl - tok0);
          __syncthreads();
          constexpr int V8 = 16 / sizeof(T);  // elements per 16-byte load
          // only the chunk's nt rows: the scores of the other rows are masked
          // out below and P V stops at nt
          for (int e = threadIdx.x; e < nt * (D / V8); e += kThreads) {
            const int i = e / (D / V8), ch = (e % (D / V8)) * V8;
            float kv[V8], vv[V8];
            const int64_t off = (int64_t)(tok0 + i) * tr.st + ch;
            load16_f32<T>(kp + off, kv);
            load16_f32<T>(vp + off, vv);
#pragma unroll
            for (int u = 0; u < V8; u += 4) {
              *reinterpret_cast<float4 *>(sK + i * (D + 4) + ch + u) = make_float4(kv[u], kv[u + 1], kv[u + 2], kv[u + 3]);
              *reinterpret_cast<float4 *>(sV + i * D + ch + u) = make_float4(vv[u], vv[u + 1], vv[u + 2], vv[u + 3]);
            }
          }
          for (int i = threadIdx.x; i < kTK; i += kThreads) sPos[i] = i < nt ? tr.pos[tok0 + i] : 0;
          __syncthreads();
          // scores of tokens lane and lane + 32 for the warp's rows (the four
          // dot products run side by side; each keeps its channel order)
          const float *q0 = sQ + (warp * kRowsPerWarp) * D;
          float s[kRowsPerWarp][2];
#pragma unroll
          for (int k = 0; k < kRowsPerWarp; ++k) s[k][0] = s[k][1] = 0.0f;
          const bool in0 = lane < nt, in1 = lane + 32 < nt;
          if (nt <= 32) {  // one token per lane (warp-uniform)
#pragma unroll 2
            for (int ch = 0; ch < D; ch += 4) {
              const float4 k0 = *reinterpret_cast<const float4 *>(sK + lane * (D + 4) + ch);
#pragma unroll
              for (int k = 0; k < kRowsPerWarp; ++k) {
                const float4 qv = *reinterpret_cast<const float4 *>(q0 + k * D + ch);
                s[k][0] = fmaf(qv.x, k0.x, s[k][0]);
                s[k][0] = fmaf(qv.y, k0.y, s[k][0]);
                s[k][0] = fmaf(qv.z, k0.z, s[k][0]);
                s[k][0] = fmaf(qv.w, k0.w, s[k][0]);
              }
            }
          } else
#pragma unroll 2
          for (int ch = 0; ch < D; ch += 4) {
            const float4 k0 = *reinterpret_cast<const float4 *>(sK + lane * (D + 4) + ch);
            const float4 k1 = *reinterpret_cast<const float4 *>(sK + (lane + 32) * (D + 4) + ch);
#pragma unroll
            for (int k = 0; k < kRowsPerWarp; ++k) {
              const float4 qv = *reinterpret_cast<const float4 *>(q0 + k * D + ch);
              s[k][0] = fmaf(qv.x, k0.x, s[k][0]);
              s[k][0] = fmaf(qv.y, k0.y, s[k][0]);
              s[k][0] = fmaf(qv.z, k0.z, s[k][0]);
              s[k][0] = fmaf(qv.w, k0.w, s[k][0]);
              s[k][1] = fmaf(qv.x, k1.x, s[k][1]);
              s[k][1] = fmaf(qv.y, k1.y, s[k][1]);
              s[k][1] = fmaf(qv.z, k1.z, s[k][1]);
              s[k][1] = fmaf(qv.w, k1.w, s[k][1]);
            }
          }
          float *pw = sP + warp * kRowsPerWarp * kTK;  // [token][row]
#pragma unroll
          for (int k = 0; k < kRowsPerWarp; ++k) {
            bool v0 = okr[k] && in0 && sPos[lane] <= qp[k], v1 = okr[k] && in1 && sPos[lane + 32] <= qp[k];
            float e0 = v0 ? exp2f(s[k][0] * b.scale_log2 - m2[k]) : 0.0f;
            float e1 = v1 ? exp2f(s[k][1] * b.scale_log2 - m2[k]) : 0.0f;
            S_c[k] += warp_sum(e0 + e1);
            n_c[k] += __popc(__ballot_sync(0xffffffffu, v0)) + __popc(__ballot_sync(0xffffffffu, v1));
            pw[lane * kRowsPerWarp + k] = e0;
            pw[(lane + 32) * kRowsPerWarp + k] = e1;
          }
          __syncwarp();
          static_assert(kRowsPerWarp == 2, "the weights of a token are read as one float2");
          for (int i = 0; i < nt; ++i) {
            const float2 p = *reinterpret_cast<const float2 *>(pw + i * kRowsPerWarp);
            float v[J];
            lds_vec<J>(sV + i * D + J * lane, v);
#pragma unroll
            for (int jj = 0; jj < J; ++jj) {
              U[0][jj] = fmaf(p.x, v[jj], U[0][jj]);
              U[1][jj] = fmaf(p.y, v[jj], U[1][jj]);
            }
          }
          __syncwarp();
        }
#pragma unroll
        for (int k = 0; k < kRowsPerWarp; ++k) {
          SE[c][k] = S_c[k];
          nE[c][k] = n_c[k];
#pragma unroll
          for (int jj = 0; jj < J; ++jj) DE[c][k][jj] = fmaf(-S_c[k], o[k][jj], U[k][jj]);
          if (c < kc && okr[k]) {
            sts_vec<J>(L.DE + ((int64_t)c * rows_full + grow[k]) * D + J * lane, DE[c][k]);
            if (lane == 0) {
              L.SE[((int64_t)c * rows_full + grow[k]) * 2] = S_c[k];
              L.SE[((int64_t)c * rows_full + grow[k]) * 2 + 1] = (float)n_c[k];
            }
          }
        }
      }

      // Eq. 6 on A u B u {E_c} for every candidate c and subset B of the
      // earlier ones, sums added in candidate order
#pragma unroll
      for (int c = 0; c < kRound; ++c) {
        if (c >= kc) break;
#pragma unroll 1
        for (int sb = 0; sb < (1 << c); ++sb) {
          float rmax = 0.0f;
#pragma unroll
          for (int k = 0; k < kRowsPerWarp; ++k) {
            float x[J], S_tot = SA[k];
            int n_tot = nA[k];
#pragma unroll
            for (int jj = 0; jj < J; ++jj) x[jj] = DA[k][jj];
#pragma unroll
            for (int bb = 0; bb < kRound - 1; ++bb) {
              if (bb < c && ((sb >> bb) & 1)) {
#pragma unroll
                for (int jj = 0; jj < J; ++jj) x[jj] += DE[bb][k][jj];
                S_tot += SE[bb][k];
                n_tot += nE[bb][k];
              }
            }
            float ss = 0.0f;
#pragma unroll
            for (int jj = 0; jj < J; ++jj) {
              float dsum = x[jj] + DE[c][k][jj];
              ss = fmaf(dsum, dsum, ss);
            }
            float num2 = warp_sum(ss);
            float rr = effect_value(n_tot + nE[c][k], nvis[k], S_tot + SE[c][k], lsum[k], num2, onorm[k]);
            if (okr[k]) rmax = fmaxf(rmax, rr);
          }
          if (lane == 0) atomicMax(reinterpret_cast<int *>(&s_rmax[combo(c, sb)]), __float_as_int(rmax));
        }
      }
      __syncthreads();
      if (threadIdx.x < kCombos && threadIdx.x < combo(kc, 0))
        atomic_max_nonneg(tab_r + G.t * kCombos + threadIdx.x, s_rmax[threadIdx.x]);
    }
    // ---------------- barrier: every block's part of the round's table is in
    if (!joint::grid_barrier(hdr, gridDim.x)) return;
    // ---------------- phase 2: replay the decisions, add the accepted sums
    for (int grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
      const Group G = decode_group(L, grp);
      const int kc = joint::round_count(L, G.t, r);
      if (kc == 0) continue;
      const unsigned acc = joint::resolve_round(tab_r + G.t * kCombos, kc, L.tau);
      if (acc == 0) continue;
#pragma unroll 1
      for (int k = 0; k < kRowsPerWarp; ++k) {
        int row = G.row0 + warp * kRowsPerWarp + k;
        if (row >= G.rows) continue;
        int64_t gr = L.row_off[G.t] + (int64_t)(G.li * b.H + G.kvh) * G.rows + row;
        float *da = L.DA + gr * D;
        float *sa = L.SA + gr * 2;
        for (int c = 0; c < kc; ++c) {
          if (!((acc >> c) & 1u)) continue;
          const float *de = L.DE + ((int64_t)c * rows_full + gr) * D;
#pragma unroll
          for (int jj = 0; jj < J; ++jj) {
            const int ch = J * lane + jj;
            da[ch] += de[ch];
          }
          if (lane == 0) {
            sa[0] += L.SE[((int64_t)c * rows_full + gr) * 2];
            sa[1] += L.SE[((int64_t)c * rows_full + gr) * 2 + 1];
          }
        }
      }
    }
    if (blockIdx.x == 0) joint::publish_round(L, r);
  }
}

template <typename T, int D>
cudaError_t launch_joint_typed(const JointLaunch &L, WsHeader *hdr, cudaStream_t s, int sm_count) {
  size_t smem = (size_t)(kRB * D + kTK * (D + 4) + kTK * D) * 4 + kTK * 4 + kWarps * kRowsPerWarp * kTK * 4;
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
  if (joint_tc_eligible(L)) return launch_joint_tc(L, hdr, stream, sm_count);
  bool bf = L.batch.dtype == COMMITKV_BF16;
  if (L.batch.d == 128)
    return bf ? launch_joint_typed<__nv_bfloat16, 128>(L, hdr, stream, sm_count)
              : launch_joint_typed<float, 128>(L, hdr, stream, sm_count);
  return bf ? launch_joint_typed<__nv_bfloat16, 64>(L, hdr, stream, sm_count)
            : launch_joint_typed<float, 64>(L, hdr, stream, sm_count);
}

int joint_rows_per_group(const JointLaunch &L) { return joint_tc_eligible(L) ? joint_tc_rows_per_group() : kRB; }
int joint_round() { return kRound; }
int joint_combos() { return kCombos; }

namespace {
__global__ void barrier_timeout_kernel(WsHeader *hdr, unsigned expected) { joint::grid_barrier(hdr, expected); }
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
