// Page deletion effects (Section 3.2, Eq. 6-8) — portable CUDA-core path.
//
// Three launches per call:
//   pass A   per (trajectory, layer, KV head, token chunk, row block):
//            online-softmax partials (max, sum, sum e*v, visible count) of
//            every probe row over the chunk;
//   combine  per probe row: merge the chunk partials into the row's final
//            max m, sum l, visible count n and output o (the stats);
//   pass B   per (trajectory, layer, KV head, page group, row block):
//            for each page E, S_E = sum_{i in E visible} e_i and
//            U_E = sum e_i v_i with e_i = exp(s_i - m), then
//            r = ||U_E - S_E o|| / ((l - S_E) ||o||)  (Eq. 6 with a = e / l),
//            max over the block's rows into R[E] and R_head[l][h][E] (Eq. 7).
// Scores are kept in base-2 units (scale * log2 e), fp32 throughout.
#include "ckv_internal.cuh"

namespace ckv {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRB = 64;               // probe rows per block
constexpr int kRowsPerWarp = kRB / kWarps;
constexpr int kTK = 64;               // tokens per shared-memory tile
constexpr float kNegInf = -__builtin_huge_valf();

__device__ __forceinline__ int find_traj(const int32_t *off, int n, int unit) {
  int t = 0;
  while (t + 1 < n && unit >= off[t + 1]) ++t;
  return t;
}

template <typename T, int D>
__device__ __forceinline__ void load_rows_q(const Batch &b, const TrajDev &tr, int l, int kvh,
                                            int row0, int rows, float *sQ) {
  const T *q = static_cast<const T *>(tr.q);
  for (int e = threadIdx.x; e < kRB * D; e += kThreads) {
    int r = e / D, c = e % D;
    float v = 0.0f;
    int row = row0 + r;
    if (row < rows) {
      int h = kvh * b.g + row / tr.W, w = row % tr.W;
      v = to_f32(q[(((int64_t)l * b.Hq + h) * tr.W + w) * D + c]);
    }
    sQ[r * D + c] = v;
  }
}

template <typename T, int D>
__device__ __forceinline__ void load_tile_kv(const TrajDev &tr, int l, int kvh, int tok0, int nt,
                                             float *sK, float *sV, int *sPos) {
  const T *kp = static_cast<const T *>(tr.k) + (int64_t)l * tr.sl + (int64_t)kvh * tr.sh;
  const T *vp = static_cast<const T *>(tr.v) + (int64_t)l * tr.sl + (int64_t)kvh * tr.sh;
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
  for (int i = threadIdx.x; i < kTK; i += kThreads) sPos[i] = i < nt ? tr.pos[tok0 + i] : 0x7fffffff;
}

__device__ __forceinline__ float dot_smem(const float *q, const float *k, int D) {
  float s = 0.0f;
#pragma unroll 8
  for (int c = 0; c < D; ++c) s = fmaf(q[c], k[c], s);
  return s;
}

// ---------------------------------------------------------------- pass A
template <typename T, int D>
__global__ void __launch_bounds__(kThreads) pass_a_kernel(const __grid_constant__ ScoreLaunch L,
                                                          float *partials) {
  extern __shared__ float smem[];
  float *sQ = smem;                       // [kRB][D]
  float *sK = sQ + kRB * D;               // [kTK][D + 1]
  float *sV = sK + kTK * (D + 1);         // [kTK][D]
  int *sPos = reinterpret_cast<int *>(sV + kTK * D);
  float *sP = reinterpret_cast<float *>(sPos + kTK);  // [kWarps][kTK]

  const Batch &b = L.batch;
  int unit = blockIdx.x;
  int t = find_traj(L.unit_off_a, b.n_traj, unit);
  const TrajDev &tr = b.t[t];
  int local = unit - L.unit_off_a[t];
  int nrb = L.nrb[t], nch = L.nchunk[t];
  int rb = local % nrb;
  local /= nrb;
  int c = local % nch;
  local /= nch;
  int kvh = local % b.H, li = local / b.H;
  int l = b.layer_ids[li];
  int rows = b.g * tr.W;
  int row0 = rb * kRB;
  int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  load_rows_q<T, D>(b, tr, l, kvh, row0, rows, sQ);

  constexpr int J = D / 32;
  float m_run[kRowsPerWarp], l_run[kRowsPerWarp], O[kRowsPerWarp][J];
  int n_run[kRowsPerWarp], qp[kRowsPerWarp];
#pragma unroll
  for (int k = 0; k < kRowsPerWarp; ++k) {
    m_run[k] = kNegInf;
    l_run[k] = 0.0f;
    n_run[k] = 0;
    int row = row0 + warp * kRowsPerWarp + k;
    qp[k] = row < rows ? tr.qpos[row % tr.W] : -0x7fffffff;
#pragma unroll
    for (int j = 0; j < J; ++j) O[k][j] = 0.0f;
  }

  int tok_begin = c * L.chunk_len;
  int tok_end = min(tr.S, tok_begin + L.chunk_len);
  for (int tok0 = tok_begin; tok0 < tok_end; tok0 += kTK) {
    int nt = min(kTK, tok_end - tok0);
    __syncthreads();
    load_tile_kv<T, D>(tr, l, kvh, tok0, nt, sK, sV, sPos);
    __syncthreads();
#pragma unroll 1
    for (int k = 0; k < kRowsPerWarp; ++k) {
      const float *q = sQ + (warp * kRowsPerWarp + k) * D;
      bool v0 = lane < nt && sPos[lane] <= qp[k], v1 = lane + 32 < nt && sPos[lane + 32] <= qp[k];
      float s0 = v0 ? dot_smem(q, sK + lane * (D + 1), D) * b.scale_log2 : kNegInf;
      float s1 = v1 ? dot_smem(q, sK + (lane + 32) * (D + 1), D) * b.scale_log2 : kNegInf;
      float mt = warp_max(fmaxf(s0, s1));
      if (mt == kNegInf) continue;  // nothing visible in this tile
      float m_new = fmaxf(m_run[k], mt);
      float alpha = exp2f(m_run[k] - m_new);
      float p0 = v0 ? exp2f(s0 - m_new) : 0.0f;
      float p1 = v1 ? exp2f(s1 - m_new) : 0.0f;
      l_run[k] = l_run[k] * alpha + warp_sum(p0 + p1);
      n_run[k] += __popc(__ballot_sync(0xffffffffu, v0)) + __popc(__ballot_sync(0xffffffffu, v1));
      m_run[k] = m_new;
      float *pw = sP + warp * kTK;
      pw[lane] = p0;
      pw[lane + 32] = p1;
      __syncwarp();
#pragma unroll
      for (int j = 0; j < J; ++j) O[k][j] *= alpha;
      for (int i = 0; i < nt; ++i) {
        float p = pw[i];
#pragma unroll
        for (int j = 0; j < J; ++j) O[k][j] = fmaf(p, sV[i * D + lane + 32 * j], O[k][j]);
      }
      __syncwarp();
    }
  }
#pragma unroll
  for (int k = 0; k < kRowsPerWarp; ++k) {
    int r = warp * kRowsPerWarp + k;
    float *dst = partials + ((int64_t)unit * kRB + r) * (D + 4);
    if (lane == 0) {
      dst[0] = m_run[k];
      dst[1] = l_run[k];
      dst[2] = (float)n_run[k];
      dst[3] = 0.0f;
    }
#pragma unroll
    for (int j = 0; j < J; ++j) dst[4 + lane + 32 * j] = O[k][j];
  }
}

// ---------------------------------------------------------------- combine
// One warp per probe row of the selected layers.
template <int D>
__global__ void __launch_bounds__(kThreads) combine_kernel(const __grid_constant__ ScoreLaunch L,
                                                           const float *partials) {
  const Batch &b = L.batch;
  int gw = (blockIdx.x * kThreads + threadIdx.x) / 32, lane = threadIdx.x % 32;
  int total = L.row_off[b.n_traj];
  if (gw >= total) return;
  int t = find_traj(L.row_off, b.n_traj, gw);
  const TrajDev &tr = b.t[t];
  int local = gw - L.row_off[t];
  int rows = b.g * tr.W;
  int row = local % rows;  // row within (layer, KV head)
  local /= rows;
  int kvh = local % b.H, li = local / b.H;
  int l = b.layer_ids[li];
  int nrb = L.nrb[t], nch = L.nchunk[t];
  int rb = row / kRB, rl = row % kRB;
  auto part = [&](int c) {
    int unit = L.unit_off_a[t] + (((li * b.H + kvh) * nch + c) * nrb + rb);
    return partials + ((int64_t)unit * kRB + rl) * (D + 4);
  };
  float m = kNegInf;
  for (int c = 0; c < nch; ++c) m = fmaxf(m, part(c)[0]);
  constexpr int J = D / 32;
  float o[J];
#pragma unroll
  for (int j = 0; j < J; ++j) o[j] = 0.0f;
  float lsum = 0.0f, n = 0.0f;
  for (int c = 0; c < nch; ++c) {
    const float *p = part(c);
    n += p[2];
    if (p[0] == kNegInf) continue;
    float a = exp2f(p[0] - m);
    lsum = fmaf(p[1], a, lsum);
#pragma unroll
    for (int j = 0; j < J; ++j) o[j] = fmaf(p[4 + lane + 32 * j], a, o[j]);
  }
  float inv = lsum > 0.0f ? 1.0f / lsum : 0.0f;
  int h = kvh * b.g + row / tr.W, w = row % tr.W;
  float *dst = L.stats[t] + (((int64_t)l * b.Hq + h) * tr.W + w) * (D + 4);
  if (lane == 0) {
    dst[0] = m == kNegInf ? m : m / 1.4426950408889634f;  // natural units
    dst[1] = lsum;
    dst[2] = n;
    dst[3] = 0.0f;
  }
#pragma unroll
  for (int j = 0; j < J; ++j) dst[4 + lane + 32 * j] = o[j] * inv;
}

// ---------------------------------------------------------------- pass B
constexpr int kPG = 16;  // pages per block

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) pass_b_kernel(const __grid_constant__ ScoreLaunch L,
                                                          WsHeader *hdr) {
  extern __shared__ float smem[];
  float *sQ = smem;
  float *sK = sQ + kRB * D;
  float *sV = sK + kTK * (D + 1);
  int *sPos = reinterpret_cast<int *>(sV + kTK * D);
  float *sP = reinterpret_cast<float *>(sPos + kTK);
  float *sR = sP + kWarps * kTK;  // [kPG] block max per page

  const Batch &b = L.batch;
  int unit = blockIdx.x;
  int t = find_traj(L.unit_off_b, b.n_traj, unit);
  const TrajDev &tr = b.t[t];
  int local = unit - L.unit_off_b[t];
  int nrb = L.nrb[t], npg = L.npg[t];
  int rb = local % nrb;
  local /= nrb;
  int pg = local % npg;
  local /= npg;
  int kvh = local % b.H, li = local / b.H;
  int l = b.layer_ids[li];
  int rows = b.g * tr.W;
  int row0 = rb * kRB;
  int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  constexpr int J = D / 32;

  load_rows_q<T, D>(b, tr, l, kvh, row0, rows, sQ);
  // this warp's rows: final stats
  float m2[kRowsPerWarp], lsum[kRowsPerWarp], onorm[kRowsPerWarp], o[kRowsPerWarp][J];
  int nvis[kRowsPerWarp], qp[kRowsPerWarp], hrow[kRowsPerWarp];
#pragma unroll
  for (int k = 0; k < kRowsPerWarp; ++k) {
    int row = row0 + warp * kRowsPerWarp + k;
    bool ok = row < rows;
    int h = kvh * b.g + (ok ? row / tr.W : 0), w = ok ? row % tr.W : 0;
    hrow[k] = ok ? h : -1;
    const float *st = L.stats[t] + (((int64_t)l * b.Hq + h) * tr.W + w) * (D + 4);
    float mn = ok ? st[0] : kNegInf;
    m2[k] = mn == kNegInf ? mn : mn * 1.4426950408889634f;
    lsum[k] = ok ? st[1] : 0.0f;
    nvis[k] = ok ? L.nvis_w[t][w] : 0;
    qp[k] = ok ? tr.qpos[w] : -0x7fffffff;
    float ss = 0.0f;
#pragma unroll
    for (int j = 0; j < J; ++j) {
      o[k][j] = ok ? st[4 + lane + 32 * j] : 0.0f;
      ss = fmaf(o[k][j], o[k][j], ss);
    }
    onorm[k] = sqrtf(warp_sum(ss));
  }

  int E0 = pg * kPG, E1 = min(tr.P, E0 + kPG);
  for (int e = threadIdx.x; e < kPG; e += kThreads) sR[e] = 0.0f;
  __syncthreads();
  for (int E = E0; E < E1; ++E) {
    int ps = tr.ps[E], pl = tr.pl[E];
    bool bad = pl < 0 || ps < 0 || ps > tr.S - pl || (E > 0 && ps < tr.ps[E - 1] + tr.pl[E - 1]);
    if (bad) {
      if (threadIdx.x == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, E);
      continue;
    }
    float S_E[kRowsPerWarp], U[kRowsPerWarp][J];
    int n_E[kRowsPerWarp];
#pragma unroll
    for (int k = 0; k < kRowsPerWarp; ++k) {
      S_E[k] = 0.0f;
      n_E[k] = 0;
#pragma unroll
      for (int j = 0; j < J; ++j) U[k][j] = 0.0f;
    }
    for (int tok0 = ps; tok0 < ps + pl; tok0 += kTK) {
      int nt = min(kTK, ps + pl - tok0);
      __syncthreads();
      load_tile_kv<T, D>(tr, l, kvh, tok0, nt, sK, sV, sPos);
      __syncthreads();
#pragma unroll 1
      for (int k = 0; k < kRowsPerWarp; ++k) {
        if (hrow[k] < 0) continue;
        const float *q = sQ + (warp * kRowsPerWarp + k) * D;
        bool v0 = lane < nt && sPos[lane] <= qp[k], v1 = lane + 32 < nt && sPos[lane + 32] <= qp[k];
        float e0 = v0 ? exp2f(dot_smem(q, sK + lane * (D + 1), D) * b.scale_log2 - m2[k]) : 0.0f;
        float e1 = v1 ? exp2f(dot_smem(q, sK + (lane + 32) * (D + 1), D) * b.scale_log2 - m2[k]) : 0.0f;
        S_E[k] += warp_sum(e0 + e1);
        n_E[k] += __popc(__ballot_sync(0xffffffffu, v0)) + __popc(__ballot_sync(0xffffffffu, v1));
        float *pw = sP + warp * kTK;
        pw[lane] = e0;
        pw[lane + 32] = e1;
        __syncwarp();
        for (int i = 0; i < nt; ++i) {
          float p = pw[i];
#pragma unroll
          for (int j = 0; j < J; ++j) U[k][j] = fmaf(p, sV[i * D + lane + 32 * j], U[k][j]);
        }
        __syncwarp();
      }
    }
    float rmax = 0.0f;
#pragma unroll
    for (int k = 0; k < kRowsPerWarp; ++k) {
      if (hrow[k] < 0) continue;
      float ss = 0.0f;
#pragma unroll
      for (int j = 0; j < J; ++j) {
        float dlt = fmaf(-S_E[k], o[k][j], U[k][j]);
        ss = fmaf(dlt, dlt, ss);
      }
      float num2 = warp_sum(ss);
      float r = effect_value(n_E[k], nvis[k], S_E[k], lsum[k], num2, onorm[k]);
      rmax = fmaxf(rmax, r);
      if (lane == 0 && L.headR[t])
        atomic_max_nonneg(L.headR[t] + ((int64_t)l * b.Hq + hrow[k]) * tr.P + E, r);
    }
    if (lane == 0) atomicMax(reinterpret_cast<int *>(sR + (E - E0)), __float_as_int(rmax));
  }
  __syncthreads();
  for (int E = E0 + threadIdx.x; E < E1; E += kThreads) atomic_max_nonneg(L.R[t] + E, sR[E - E0]);
}

// Per trajectory and window position w: the number of resident tokens with
// pos <= qpos[w] (positions increase, so a binary search).
__global__ void __launch_bounds__(256) count_visible_kernel(const __grid_constant__ ScoreLaunch L) {
  const int t = blockIdx.x;
  const TrajDev &tr = L.batch.t[t];
  for (int w = threadIdx.x; w < tr.W; w += blockDim.x) {
    const int qp = tr.qpos[w];
    int a = 0, b = tr.S;
    while (a < b) {
      int mid = (a + b) >> 1;
      if (tr.pos[mid] <= qp) a = mid + 1;
      else b = mid;
    }
    L.nvis_w[t][w] = a;
  }
}

template <typename T, int D>
cudaError_t launch_typed(const ScoreLaunch &L, float *partials, WsHeader *hdr, cudaStream_t s) {
  size_t smem = (size_t)(kRB * D + kTK * (D + 1) + kTK * D) * 4 + kTK * 4 + kWarps * kTK * 4 + kPG * 4;
  cudaError_t e;
  e = cudaFuncSetAttribute(pass_a_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(pass_b_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  count_visible_kernel<<<L.batch.n_traj, 256, 0, s>>>(L);
  int na = L.from_stats ? 0 : L.unit_off_a[L.batch.n_traj];
  if (na > 0) pass_a_kernel<T, D><<<na, kThreads, smem, s>>>(L, partials);
  int rows = L.from_stats ? 0 : L.row_off[L.batch.n_traj];
  if (rows > 0) combine_kernel<D><<<(rows * 32 + kThreads - 1) / kThreads, kThreads, 0, s>>>(L, partials);
  int nb = L.unit_off_b[L.batch.n_traj];
  if (nb > 0) pass_b_kernel<T, D><<<nb, kThreads, smem, s>>>(L, hdr);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score_simt(const ScoreLaunch &L, float *partials, WsHeader *hdr,
                              cudaStream_t stream) {
  bool bf = L.batch.dtype == COMMITKV_BF16;
  if (L.batch.d == 128)
    return bf ? launch_typed<__nv_bfloat16, 128>(L, partials, hdr, stream)
              : launch_typed<float, 128>(L, partials, hdr, stream);
  return bf ? launch_typed<__nv_bfloat16, 64>(L, partials, hdr, stream)
            : launch_typed<float, 64>(L, partials, hdr, stream);
}

int simt_rows_per_block() { return kRB; }
int simt_pages_per_block() { return kPG; }

}  // namespace ckv
