// Pieces of the greedy joint test (Section 3.3, Eq. 11) shared by its two
// kernels (CUDA-core and tensor-core): the round structure, the grid
// barrier of the cooperative launch and the replay of a round's decisions.
//
// Candidates are taken in rounds of kRound.  For every candidate c of a
// round and every subset B of the round's earlier candidates, Eq. 6 is
// evaluated on A u B u {E_c} (A = the pages accepted in earlier rounds),
// with the sums added in candidate order, and the max over rows (Eq. 7)
// goes to a per-round table slot combo(c, B).  After the barrier the
// decisions are replayed from the table: candidate c is accepted iff its
// value for B = the round's candidates accepted before it is <= tau.  The
// slot of (c, B) is T - 1 with T = B u {c} as a bit set, so the 15 slots of
// a round of four are its 15 non-empty subsets.
#pragma once

#include "ckv_internal.cuh"

namespace ckv {
namespace joint {

constexpr int kRound = 4;                   // candidates per round
constexpr int kCombos = (1 << kRound) - 1;  // (candidate, subset of the earlier ones) pairs
constexpr uint64_t kWaitNs = 1000000000ull;  // 1 s per barrier

static_assert(kRound * 4 <= 32, "accepted masks travel in one word");

// Table slot of candidate c with the subset s of candidates 0..c-1.
__host__ __device__ constexpr int combo(int c, int s) { return (1 << c) - 1 + s; }

__device__ __forceinline__ int find_group_traj(const int32_t *off, int n, int unit) {
  int t = 0;
  while (t + 1 < n && unit >= off[t + 1]) ++t;
  return t;
}

// Sense-free generation barrier over all blocks of a cooperative launch,
// with a bounded wait.  Returns false (and records a timeout) on expiry or
// when another block has aborted.
__device__ inline bool grid_barrier(WsHeader *hdr, unsigned nblocks) {
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

// Number of rounds of the launch (the longest candidate list).
__device__ __forceinline__ int round_total(const JointLaunch &L) {
  int rounds = 0;
  for (int t = 0; t < L.batch.n_traj; ++t) {
    int nc = min(max(L.n_cand[t], 0), L.batch.t[t].P);
    rounds = max(rounds, (nc + kRound - 1) / kRound);
  }
  return rounds;
}

// Candidates of round r for trajectory t (0 when the scan is over).
__device__ __forceinline__ int round_count(const JointLaunch &L, int t, int r) {
  int nc = min(max(L.n_cand[t], 0), L.batch.t[t].P);
  return max(0, min(kRound, nc - r * kRound));
}

// The round's decisions, replayed from its table: bit c set = accepted.
__device__ __forceinline__ unsigned resolve_round(const float *tab, int kc, float tau) {
  unsigned acc = 0;
  for (int c = 0; c < kc; ++c) {
    float R = *(volatile const float *)(tab + combo(c, acc));
    if (R <= tau) acc |= 1u << c;
  }
  return acc;
}

// Table of round r (three rotate: r is being filled, r - 1 is read after
// the barrier, r + 2 is cleared).
__device__ __forceinline__ float *round_table(const JointLaunch &L, int r) {
  return L.roundR + (size_t)(r % 3) * L.batch.n_traj * kCombos;
}

// After round r's barrier, by one block: the step values and accepted
// pages of the round, and the table of round r + 2 cleared (its last reads
// were before this round's barrier).
__device__ __forceinline__ void publish_round(const JointLaunch &L, int r) {
  const Batch &b = L.batch;
  for (int t = threadIdx.x; t < b.n_traj; t += blockDim.x) {
    const int kc = round_count(L, t, r);
    const float *tab = round_table(L, r) + t * kCombos;
    unsigned acc = 0;
    for (int c = 0; c < kc; ++c) {
      const int j = r * kRound + c;
      const int E = L.cand[t][j];
      const float R = *(volatile const float *)(tab + combo(c, acc));
      if (L.stepR_out[t]) L.stepR_out[t][j] = R;
      if (R <= L.tau) {
        acc |= 1u << c;
        if (E >= 0 && E < b.t[t].P) L.accepted[t][E] = 1;
      }
    }
    float *next = round_table(L, r + 2) + t * kCombos;
    for (int i = 0; i < kCombos; ++i) next[i] = 0.0f;
  }
}

}  // namespace joint
}  // namespace ckv
