// Internal declarations of the CommitKV CUDA library (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "commitkv.h"

namespace ckv {

constexpr int kMaxTraj = COMMITKV_MAX_TRAJ;
constexpr int kMaxLayers = 256;

// Per-trajectory view, copied into kernel parameters.
struct TrajDev {
  const void *k, *v;
  int64_t sl, sh, st;  // strides in elements
  const int32_t *pos;
  const void *q;
  const int32_t *qpos;
  const int32_t *ps, *pl;
  int32_t S, W, P, pad;
};

// A batch of trajectories sharing one model shape.
struct Batch {
  int32_t n_traj, M, H, Hq, g, d, dtype, n_layers;
  float scale;       // softmax scale (natural exponent)
  float scale_log2;  // scale * log2(e): scores are kept in base-2 units
  uint8_t layer_ids[kMaxLayers];  // selected layers, in order
  TrajDev t[kMaxTraj];
};

// Workspace header (first 256 bytes of every workspace).
struct WsHeader {
  int32_t status;           // first device-side error (commitkv_status), 0 = none
  int32_t abort;            // set when a bounded wait gave up
  uint32_t bar_count;       // grid barrier arrivals
  uint32_t bar_gen;         // grid barrier generation
  int32_t err_info[4];      // where the first error was seen (debug)
  uint32_t pad[56];
};
static_assert(sizeof(WsHeader) == 256, "workspace header is 256 bytes");

__device__ __forceinline__ void record_error(WsHeader *h, int code, int info = 0) {
  if (atomicCAS(&h->status, 0, code) == 0) h->err_info[0] = info;
}

// Non-negative floats order like their bit patterns: max via integer atomics.
__device__ __forceinline__ void atomic_max_nonneg(float *addr, float v) {
  atomicMax(reinterpret_cast<int *>(addr), __float_as_int(v));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Deletion-effect value of one probe row for a deleted token set, from
// unnormalised sums with the row's final max (Eq. 6 with a_i = e_i / l):
//   num2 = ||U_del - S_del * o||^2,  r = sqrt(num2) / ((l - S_del) * ||o||)
// with the degenerate rules: nothing visible deleted -> 0; everything
// visible deleted (or no visible mass left) -> inf; ||o|| = 0 -> 0 or inf.
__device__ __forceinline__ float effect_value(int n_del, int n_vis, float S_del, float l,
                                              float num2, float onorm) {
  if (n_del == 0) return 0.0f;
  if (n_del >= n_vis) return __int_as_float(0x7f800000);
  if (onorm == 0.0f) return num2 == 0.0f ? 0.0f : __int_as_float(0x7f800000);
  float rest = l - S_del;
  if (!(rest > 0.0f)) return __int_as_float(0x7f800000);
  return sqrtf(num2) / (rest * onorm);
}

// Host-side argument checks (api.cu), shared by every entry point that
// takes these arguments so that they refuse the same inputs.
commitkv_status check_shape(const commitkv_shape *s);
commitkv_status check_trajs(const commitkv_shape *s, int n_traj, const commitkv_traj *tr, bool need_q);
commitkv_status check_compact_args(const commitkv_shape *s, int32_t n_traj, const commitkv_traj *tr,
                                   const uint8_t *const *retired, const int32_t *const *pending,
                                   const int32_t *n_pending, const float *const *pending_priority,
                                   const float *const *fill_score, int32_t budget_B,
                                   int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                   int32_t *const *idx_out, const int32_t *n_idx_out);

// Launch helpers implemented in the .cu files ------------------------------

struct ScoreLaunch {
  Batch batch;
  int32_t unit_off_a[kMaxTraj + 1];  // pass A unit offsets per trajectory
  int32_t unit_off_b[kMaxTraj + 1];  // pass B unit offsets per trajectory
  int32_t nchunk[kMaxTraj];
  int32_t nrb[kMaxTraj];             // row blocks per (layer, KV head)
  int32_t npg[kMaxTraj];             // page groups per (layer, KV head)
  int32_t row_off[kMaxTraj + 1];     // stats row offsets (selected layers only)
  int32_t chunk_len;
  float *stats[kMaxTraj];            // [M][Hq][W][d + 4]
  float *R[kMaxTraj];
  float *headR[kMaxTraj];
  int32_t *nvis_w[kMaxTraj];         // [W]: resident tokens visible to each window position
  int32_t from_stats;                // the stats are the caller's: no flash pass, no combine
};

cudaError_t launch_score_simt(const ScoreLaunch &L, float *partials, WsHeader *hdr,
                              cudaStream_t stream);

struct ClassifyLaunch {
  int32_t n_traj;
  int32_t P[kMaxTraj];
  const float *Rm[kMaxTraj];
  const float *Rp[kMaxTraj];
  const uint8_t *el[kMaxTraj];
  uint8_t *state[kMaxTraj];
  int32_t *cand[kMaxTraj];
  int32_t *scratch[kMaxTraj];  // [P_t] ints
  int32_t *n_cand;
  float tau_use, tau_dead;
  double rho_use, rho_dead;
  uint32_t variant;  // COMMITKV_CLASSIFY_NO_* bits (the ablations of Section 4.4)
};
cudaError_t launch_classify(const ClassifyLaunch &L, WsHeader *hdr, cudaStream_t stream);

struct JointLaunch {
  Batch batch;
  int32_t group_off[kMaxTraj + 1];  // row groups per trajectory (prefix)
  int32_t nrb[kMaxTraj];
  const float *stats[kMaxTraj];
  const int32_t *cand[kMaxTraj];
  const int32_t *n_cand;
  uint8_t *accepted[kMaxTraj];
  float *stepR_out[kMaxTraj];
  float *DA;                // workspace [rows_full][d]: D_A of every row
  float *DE;                // workspace [round][rows_full][d]: D_c of the round's candidates
  float *SA;                // workspace [rows_full][2]: S_A, n_A
  float *SE;                // workspace [round][rows_full][2]: S_c, n_c
  float *roundR;            // workspace [3][n_traj][combos]: per-round tables of row maxima
  int64_t rows_full;        // rows of all layers, the stride of DE and SE
  int32_t row_off[kMaxTraj + 1];
  float tau;
};
// Tensor-core kernel (bf16, head_dim 128, 16-byte aligned rows) when the
// launch allows it, else the CUDA-core kernel; the row-group size follows.
cudaError_t launch_joint(const JointLaunch &L, WsHeader *hdr, cudaStream_t stream, int sm_count);
int joint_rows_per_group(const JointLaunch &L);
bool joint_tc_eligible(const JointLaunch &L);
int joint_tc_rows_per_group();
cudaError_t launch_joint_tc(const JointLaunch &L, WsHeader *hdr, cudaStream_t stream, int sm_count);
int joint_round();   // candidates per round
int joint_combos();  // (candidate, earlier subset) pairs per round

struct CompactLaunch {
  int32_t n_traj, M, H, d, elem_bytes;
  TrajDev t[kMaxTraj];
  const uint8_t *retired[kMaxTraj];
  const int32_t *pending[kMaxTraj];
  int32_t n_pending[kMaxTraj];
  const float *prio[kMaxTraj];
  const float *fill[kMaxTraj];
  uint8_t *cls[kMaxTraj];     // workspace [S_t]
  int32_t *idx[kMaxTraj];
  int32_t *n_idx;
  void *k_out[kMaxTraj];
  void *v_out[kMaxTraj];
  int32_t *pos_out[kMaxTraj];
  int32_t B, B_N, cap;
  int32_t in_place;  // gather into the cache itself (rows 0..|I|-1 of every slice)
};
cudaError_t launch_compact(const CompactLaunch &L, WsHeader *hdr, cudaStream_t stream);

}  // namespace ckv
