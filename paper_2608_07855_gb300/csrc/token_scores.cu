// Per-token window-attention scores for the fill of the remaining budget at
// a compression checkpoint (Eq. 13): token i scores
//     max over selected layers l, query heads h and window positions p that
//     see it (pos_i <= qpos_p) of  a_{p,i} = exp(s_{p,i} - m_p) / l_p,
// 0 if no window position sees it; s = softmax_scale <q_p, k_i>, and m_p,
// l_p are the row statistics of the same cache and window (the stats_out of
// commitkv_page_effects).  The paper defers its fill rule to an appendix it
// does not include; this is window attention in the spirit of SnapKV, whose
// probe windows the paper builds on.
//
// Tensor-core path (bf16, head_dim 128, 16-byte aligned rows): a persistent
// kernel, one CTA of 320 threads per SM, items (trajectory, layer, KV head,
// token chunk, 128-row tile of probe rows), the row tiles of one chunk
// adjacent so that their K re-reads hit L2.  Per 128-token tile of K:
//   warp 0  TMA: Q tile once per item, K tiles through a 4-stage ring
//   warp 1  D[token][row] = K Q^T (tcgen05, fp32 in TMEM, two buffers)
//   warps 2..9  two groups of four taking alternate tiles, one thread per
//           token (TMEM lane): for every row p, 2^(s c - m_p log2 e -
//           log2 l_p) on the rows that see the token (all of them for the
//           tokens at or before the smallest window position), max, and one
//           atomic max into the token's score.
// K rows are the MMA's M operand, so each thread reads its own token's row
// of scores and the max over probe rows needs no cross-thread reduction.
// CUDA-core path (fp32, head_dim 64, other layouts): one thread per token,
// the probe rows of a slice staged in shared memory.
// Every wait is bounded (1 s); on expiry the kernel records
// COMMITKV_ERR_TIMEOUT and returns.
#include <cudaTypedefs.h>
#include <string.h>

#include "ckv_internal.cuh"
#include "score_tc.cuh"
#include "sm103.cuh"

namespace ckv {
namespace ts {
namespace {

using namespace ckv::sm103;

constexpr int D = 128;
constexpr int BT = 128;  // tokens per tile (MMA M)
constexpr int BR = 128;  // probe rows per tile (MMA N)
constexpr int NST = 4;   // K stages
constexpr int kTilesPerItem = 16;
constexpr uint64_t kWait = 1000000000ull;
constexpr uint32_t kTileBytes = BT * D * 2;
constexpr uint32_t kHalf = kTileBytes / 2;

struct TsTraj {
  const int32_t *pos, *qpos;
  const float *stats;  // [M][Hq][W][D + 4]
  float *score;        // [S]
  int S, W, nrt, nchunk;
};

struct TsLaunch {
  tc::TcMaps maps[tc::kMaxTc];
  TsTraj t[tc::kMaxTc];
  int n_traj, M, H, Hq, g, n_layers;
  float scale_log2;
  int item_off[tc::kMaxTc + 1];
  uint8_t layer_ids[kMaxLayers];
};

struct Item {
  int t, l, li, kvh, rt, c;
};

__device__ __forceinline__ Item decode(const TsLaunch &L, int item) {
  Item it;
  it.t = 0;
  while (it.t + 1 < L.n_traj && item >= L.item_off[it.t + 1]) ++it.t;
  const TsTraj &tr = L.t[it.t];
  int local = item - L.item_off[it.t];
  it.rt = local % tr.nrt;
  local /= tr.nrt;
  it.c = local % tr.nchunk;
  local /= tr.nchunk;
  it.kvh = local % L.H;
  it.li = local / L.H;
  it.l = L.layer_ids[it.li];
  return it;
}

__device__ __forceinline__ uint64_t desc_kmajor(const uint8_t *tile, int ks) {
  return smem_desc(smem_addr(tile) + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024, kSwizzle128B);
}

__device__ __forceinline__ void tma4(void *dst, const CUtensorMap *m, int x, int tok, int h, int l, uint64_t *bar,
                                     uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(tok), "r"(h), "r"(l), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

struct Smem {
  alignas(1024) uint8_t q[kTileBytes];
  alignas(1024) uint8_t k[NST][kTileBytes];
  // per epilogue warp: its own copy of the item's row terms (no cross-warp barrier)
  float mlog[8][BR];  // row max + log2(row sum), base 2; +inf: the row sees nothing
  int qp[8][BR];      // window position of the row
  uint64_t q_full, q_empty, k_full[NST], k_empty[NST], d_full[2], d_empty[2], drain;
  uint32_t tmem;
  int abort_flag;
};

__global__ void __launch_bounds__(320, 1) token_scores_tc(const __grid_constant__ TsLaunch L, WsHeader *hdr) {
  extern __shared__ uint8_t smem_raw[];
  Smem &sm = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n_items = L.item_off[L.n_traj];
  volatile int *abort_flag = &sm.abort_flag;
  if (threadIdx.x == 0) {
    sm.abort_flag = 0;
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, 1);
    for (int s = 0; s < NST; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.d_full[b], 1);
      mbar_init(&sm.d_empty[b], 4);
    }
    mbar_init(&sm.drain, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_normal();
      uint32_t g = 0, n_local = 0, n_k = 0;
      bool stop = false;
      for (int item = blockIdx.x; item < n_items && !stop; item += gridDim.x, ++n_local) {
        if (*abort_flag) break;
        const Item a = decode(L, item);
        const TsTraj &tr = L.t[a.t];
        const tc::TcMaps &mp = L.maps[a.t];
        if (n_local > 0 && !mbar_wait(&sm.q_empty, (n_local - 1) & 1, kWait, abort_flag)) break;
        mbar_expect_tx(&sm.q_full, kTileBytes);
        const int qrow = (a.l * L.Hq + a.kvh * L.g) * tr.W + a.rt * BR;
        tma_load_2d(sm.q, &mp.q, 0, qrow, &sm.q_full, pol);
        tma_load_2d(sm.q + kHalf, &mp.q, 64, qrow, &sm.q_full, pol);
        const int t0 = a.c * kTilesPerItem * BT, t1 = min(tr.S, t0 + kTilesPerItem * BT);
        for (int tok = t0; tok < t1; tok += BT, ++g) {
          const int s = g % NST;
          if (g >= NST && !mbar_wait(&sm.k_empty[s], ((g / NST) - 1) & 1, kWait, abort_flag)) {
            stop = true;
            break;
          }
          mbar_expect_tx(&sm.k_full[s], kTileBytes);
          tma4(sm.k[s], &mp.k, 0, tok, a.kvh, a.l, &sm.k_full[s], pol);
          tma4(sm.k[s] + kHalf, &mp.k, 64, tok, a.kvh, a.l, &sm.k_full[s], pol);
          ++n_k;
        }
      }
      if (*abort_flag) {
        // let the copies already issued land before the CTA leaves
        for (uint32_t u = (n_k > NST ? n_k - NST : 0); u < n_k; ++u)
          mbar_wait_drain(&sm.k_full[u % NST], (u / NST) & 1, kWait);
        if (n_local > 0) mbar_wait_drain(&sm.q_full, (n_local - 1) & 1, kWait);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(BT, BR, 0, 0);
      uint32_t g = 0, n_local = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x, ++n_local) {
        const Item a = decode(L, item);
        const TsTraj &tr = L.t[a.t];
        const int t0 = a.c * kTilesPerItem * BT, t1 = min(tr.S, t0 + kTilesPerItem * BT);
        const int ntile = (t1 - t0 + BT - 1) / BT;
        if (!mbar_wait(&sm.q_full, n_local & 1, kWait, abort_flag)) break;
        tc_fence_after();
        for (int j = 0; j < ntile; ++j, ++g) {
          const int s = g % NST, b = g & 1;
          if (!mbar_wait(&sm.k_full[s], (g / NST) & 1, kWait, abort_flag) ||
              (g >= 2 && !mbar_wait(&sm.d_empty[b], ((g >> 1) - 1) & 1, kWait, abort_flag))) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks)
            mma_bf16(tm + b * BR, desc_kmajor(sm.k[s], ks), desc_kmajor(sm.q, ks), idesc, ks > 0);
          mma_commit(&sm.d_full[b]);
          mma_commit(&sm.k_empty[s]);
          if (j + 1 == ntile) mma_commit(&sm.q_empty);
        }
      }
      if (*abort_flag) {
        mma_commit(&sm.drain);  // every MMA issued by this thread has completed
        mbar_wait_drain(&sm.drain, 0, kWait);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (warps 2..9)
    // Two groups of four warps take alternate tiles (group 0 the even
    // tiles in TMEM buffer 0, group 1 the odd ones in buffer 1).
    const int ew = warp - 2;          // this warp's copy of the row terms
    const int hb = ew >> 2;           // this group's tiles: g & 1 == hb
    const int wq = warp & 3;          // TMEM lane quarter: warps 2..5 -> 2, 3, 0, 1; 6..9 -> 2, 3, 0, 1
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    float *mlog = sm.mlog[ew];
    int *qp = sm.qp[ew];
    uint32_t g = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const Item a = decode(L, item);
      const TsTraj &tr = L.t[a.t];
      const int rows = L.g * tr.W;
      // e = 2^(s c - m log2 e - log2 l) = exp(s - m) / l; every row that
      // sees anything sees the tokens at or before the smallest window
      // position, which then need no per-row test
      __syncwarp();
      int qmin = 0x7fffffff;
      for (int r = lane; r < BR; r += 32) {
        const int row = a.rt * BR + r;
        float ml = INFINITY;
        int q = 0x7fffffff;
        if (row < rows) {
          const int h = a.kvh * L.g + row / tr.W, w = row % tr.W;
          const float4 st = *reinterpret_cast<const float4 *>(tr.stats + (((int64_t)a.l * L.Hq + h) * tr.W + w) *
                                                                           (D + 4));
          if (st.y > 0.0f && st.x != -INFINITY) {  // a row that sees nothing scores no token
            ml = fmaf(st.x, 1.4426950408889634f, log2f(st.y));
            q = tr.qpos[w];
          }
        }
        mlog[r] = ml;
        qp[r] = q;
        qmin = min(qmin, q);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) qmin = min(qmin, __shfl_xor_sync(0xffffffffu, qmin, o));
      __syncwarp();
      const int t0 = a.c * kTilesPerItem * BT, t1 = min(tr.S, t0 + kTilesPerItem * BT);
      for (int tok0 = t0; tok0 < t1; tok0 += BT, ++g) {
        const int b = g & 1;
        if (b != hb) continue;
        const int i = tok0 + wq * 32 + lane;  // this thread's token
        const bool valid = i < t1;
        const int pi = valid ? tr.pos[i] : 0x7fffffff;
        const bool seen_by_all = pi <= qmin;
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.d_full[b], (g >> 1) & 1, kWait, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        float best = 0.0f;
#pragma unroll 1
        for (int c0 = 0; c0 < BR; c0 += 32) {
          float x[32];
          tmem_ld32f(tm + lane_base + b * BR + c0, x);
          tmem_wait_ld();
          if (__all_sync(0xffffffffu, seen_by_all)) {
#pragma unroll
            for (int r = 0; r < 32; ++r) best = fmaxf(best, fast_exp2(fmaf(x[r], L.scale_log2, -mlog[c0 + r])));
          } else {
#pragma unroll
            for (int r = 0; r < 32; ++r) {
              const float e = fast_exp2(fmaf(x[r], L.scale_log2, -mlog[c0 + r]));
              best = pi <= qp[c0 + r] ? fmaxf(best, e) : best;
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.d_empty[b]);
        if (valid && best > 0.0f) atomic_max_nonneg(tr.score + i, best);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tm, 256);
  if (threadIdx.x == 0 && sm.abort_flag) record_error(hdr, COMMITKV_ERR_TIMEOUT, 20);
}

// ---------------------------------------------------------------- CUDA cores
constexpr int kSimtThreads = 128;  // one token per thread
constexpr int kSimtRows = 32;      // probe rows staged at a time

struct SimtLaunch {
  Batch B;
  const float *stats[kMaxTraj];
  float *score[kMaxTraj];
  int32_t blk_off[kMaxTraj + 1];
};

template <typename T, int DD>
__global__ void __launch_bounds__(kSimtThreads) token_scores_simt(const __grid_constant__ SimtLaunch S) {
  const Batch &B = S.B;
  const int32_t *blk_off = S.blk_off;
  int t = 0;
  while (t + 1 < B.n_traj && (int)blockIdx.x >= blk_off[t + 1]) ++t;
  const TrajDev &tr = B.t[t];
  int local = blockIdx.x - blk_off[t];
  const int nch = (tr.S + kSimtThreads - 1) / kSimtThreads;
  const int ch = local % nch;
  local /= nch;
  const int kvh = local % B.H, li = local / B.H, l = B.layer_ids[li];
  const int i = ch * kSimtThreads + threadIdx.x;
  const bool valid = i < tr.S;
  __shared__ float sq[kSimtRows][DD];
  __shared__ float sm2[kSimtRows], sil[kSimtRows];
  __shared__ int sqp[kSimtRows];
  float k[DD];
  const T *kp = static_cast<const T *>(tr.k) + (int64_t)l * tr.sl + (int64_t)kvh * tr.sh + (int64_t)i * tr.st;
#pragma unroll
  for (int c = 0; c < DD; ++c) k[c] = valid ? to_f32(kp[c]) : 0.0f;
  const int pi = valid ? tr.pos[i] : 0x7fffffff;
  const int rows = B.g * tr.W;
  const T *q = static_cast<const T *>(tr.q);
  float best = 0.0f;
  for (int r0 = 0; r0 < rows; r0 += kSimtRows) {
    __syncthreads();
    for (int e = threadIdx.x; e < kSimtRows * DD; e += kSimtThreads) {
      const int r = e / DD, c = e % DD, row = r0 + r;
      float v = 0.0f;
      if (row < rows) {
        const int h = kvh * B.g + row / tr.W, w = row % tr.W;
        v = to_f32(q[(((int64_t)l * B.Hq + h) * tr.W + w) * DD + c]);
      }
      sq[r][c] = v;
    }
    for (int r = threadIdx.x; r < kSimtRows; r += kSimtThreads) {
      const int row = r0 + r;
      float mm = -INFINITY, il = 0.0f;
      int qq = -0x7fffffff - 1;
      if (row < rows) {
        const int h = kvh * B.g + row / tr.W, w = row % tr.W;
        const float *st = S.stats[t] + (((int64_t)l * B.Hq + h) * tr.W + w) * (DD + 4);
        if (st[1] > 0.0f && st[0] != -INFINITY) {
          mm = st[0] * 1.4426950408889634f;
          il = 1.0f / st[1];
          qq = tr.qpos[w];
        }
      }
      sm2[r] = mm;
      sil[r] = il;
      sqp[r] = qq;
    }
    __syncthreads();
    for (int r = 0; r < kSimtRows && r0 + r < rows; ++r) {
      if (pi > sqp[r]) continue;
      float dot = 0.0f;
#pragma unroll
      for (int c = 0; c < DD; ++c) dot = fmaf(k[c], sq[r][c], dot);
      best = fmaxf(best, exp2f(fmaf(dot, B.scale_log2, -sm2[r])) * sil[r]);
    }
  }
  if (valid && best > 0.0f) atomic_max_nonneg(S.score[t] + i, best);
}

}  // namespace

size_t smem_bytes() { return sizeof(Smem) + 1024; }

// Launches the tensor-core kernel over the trajectories of `b` (at most
// tc::kMaxTc per launch).
cudaError_t launch_tc(const Batch &b, const float *const *stats, float *const *score, WsHeader *hdr,
                      cudaStream_t s, int sm_count) {
  static thread_local TsLaunch L;
  cudaError_t e = cudaFuncSetAttribute(token_scores_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_bytes());
  if (e != cudaSuccess) return e;
  for (int b0 = 0; b0 < b.n_traj; b0 += tc::kMaxTc) {
    const int nb = b.n_traj - b0 < tc::kMaxTc ? b.n_traj - b0 : tc::kMaxTc;
    memset(&L, 0, sizeof L);
    L.n_traj = nb;
    L.M = b.M;
    L.H = b.H;
    L.Hq = b.Hq;
    L.g = b.g;
    L.n_layers = b.n_layers;
    L.scale_log2 = b.scale_log2;
    memcpy(L.layer_ids, b.layer_ids, sizeof L.layer_ids);
    for (int i = 0; i < nb; ++i) {
      const TrajDev &x = b.t[b0 + i];
      TsTraj &tt = L.t[i];
      tt.pos = x.pos;
      tt.qpos = x.qpos;
      tt.stats = stats[b0 + i];
      tt.score = score[b0 + i];
      tt.S = x.S;
      tt.W = x.W;
      tt.nrt = (b.g * x.W + BR - 1) / BR;
      tt.nchunk = (x.S + kTilesPerItem * BT - 1) / (kTilesPerItem * BT);
      const bool active = x.S > 0 && x.W > 0;
      L.item_off[i + 1] = L.item_off[i] + (active ? b.n_layers * b.H * tt.nchunk * tt.nrt : 0);
      if (active && !tc::build_maps(L.maps[i], x, b.M, b.H, b.Hq)) return cudaErrorInvalidValue;
    }
    const int n = L.item_off[nb];
    if (n > 0) token_scores_tc<<<n < sm_count ? n : sm_count, 320, smem_bytes(), s>>>(L, hdr);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// The CUDA-core kernel over every trajectory of `b` in one launch.
cudaError_t launch_simt(const Batch &b, const float *const *stats, float *const *score, cudaStream_t s) {
  static thread_local SimtLaunch S;
  memset(&S, 0, sizeof S);
  S.B = b;
  for (int t = 0; t < b.n_traj; ++t) {
    const TrajDev &x = b.t[t];
    S.stats[t] = stats[t];
    S.score[t] = score[t];
    const int nch = (x.S + kSimtThreads - 1) / kSimtThreads;
    S.blk_off[t + 1] = S.blk_off[t] + (x.S > 0 && x.W > 0 ? b.n_layers * b.H * nch : 0);
  }
  const int n = S.blk_off[b.n_traj];
  if (n <= 0) return cudaSuccess;
  if (b.dtype == COMMITKV_BF16) {
    if (b.d == 128) token_scores_simt<__nv_bfloat16, 128><<<n, kSimtThreads, 0, s>>>(S);
    else token_scores_simt<__nv_bfloat16, 64><<<n, kSimtThreads, 0, s>>>(S);
  } else {
    if (b.d == 128) token_scores_simt<float, 128><<<n, kSimtThreads, 0, s>>>(S);
    else token_scores_simt<float, 64><<<n, kSimtThreads, 0, s>>>(S);
  }
  return cudaGetLastError();
}

}  // namespace ts
}  // namespace ckv
