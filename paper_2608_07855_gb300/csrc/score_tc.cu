// Page deletion effects (Section 3.2, Eq. 6-8) on the 5th-generation tensor
// cores: bf16 K/V/Q, head_dim 128, fp32 accumulation in tensor memory.
//
//   pass A   persistent, warp-specialised flash forward over 128-token tiles
//            of a token chunk: S = Q K^T (tcgen05, TMEM), online softmax in
//            base 2 with a lazy max (O in TMEM is rescaled only when the row
//            max grows by more than 2^8), O += P V (tcgen05); writes the
//            chunk's (max, sum, count, O) per probe row.
//   combine  merges a slice's chunk partials into the row stats
//            (m, l, n, o) of the whole cache.
//   slots    per trajectory, the prefix count of 16-token slots per page.
//   pass B   persistent, over tiles of 8 slots: every page is loaded as
//            16-row TMA boxes into slots of its own, so one page's columns
//            never share a 16-wide MMA k-block with another page.
//            S = Q K_slots^T; e = exp(s - m) on the page's visible tokens;
//            U_E = sum_{i in E} e_i v_i by per-slot MMAs accumulating into
//            one of two 128-column TMEM accumulators; a separate epilogue
//            warpgroup reduces U_E to
//              r = ||U_E - S_E o|| / ((l - S_E) ||o||)      (Eq. 6 with a = e / l)
//            and max-reduces r over rows into R[E] (Eq. 7).
// Every mbarrier wait is bounded (1 s); on expiry the kernel records
// COMMITKV_ERR_TIMEOUT and all warps leave their loops.
#include <cudaTypedefs.h>
#include <stdlib.h>

#include "ckv_internal.cuh"
#include "sm103.cuh"
#include "score_tc.cuh"

namespace ckv {
namespace tc {
namespace {

using namespace ckv::sm103;

constexpr int D = 128;
constexpr int BM = 128;  // probe rows per tile (MMA M)
constexpr int BT = 128;  // KV rows per tile (MMA N of Q K^T, K of P V)
constexpr int NKB = 3;   // pass B: K stages (with their slot tables)
constexpr int NVB = 2;   // pass B: V stages
constexpr int SLOT = 16;
constexpr int SLOTS = BT / SLOT;  // slots per pass-B tile
constexpr int NFIFO = 16;         // page-sum FIFO depth (>= 2 x SLOTS)
constexpr uint64_t kWait = 1000000000ull;
constexpr float kLazy = 8.0f;     // rescale O when the max grows by > 2^8
constexpr int kRing = kPartialRing;  // partial slots per flash CTA of the fused launch

constexpr uint32_t kTileBytes = BT * D * 2;  // 32 KB (two 16 KB halves)
constexpr uint32_t kHalf = kTileBytes / 2;

// ----------------------------------------------------------------- helpers
__device__ __forceinline__ int traj_of(const int32_t *off, int n, int item) {
  int t = 0;
  while (t + 1 < n && item >= off[t + 1]) ++t;
  return t;
}

__device__ __forceinline__ void tma4(void *dst, const CUtensorMap *m, int x, int tok, int h, int l,
                                     uint64_t *bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(tok), "r"(h), "r"(l), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}


// K-major operand tile (rows x 128 elements, two 64-element halves): the
// descriptor of the 16-element k-step `ks`.
__device__ __forceinline__ uint64_t desc_kmajor(const uint8_t *tile, int ks) {
  return smem_desc(smem_addr(tile) + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024, kSwizzle128B);
}
// MN-major B operand (V rows = k, 128 channels = n): k-step of 16 rows.
__device__ __forceinline__ uint64_t desc_v(const uint8_t *tile, int ks) {
  return smem_desc(smem_addr(tile) + ks * 2048, kHalf, 1024, kSwizzle128B);
}

// ============================================================== fused-launch plumbing
// Partial slot of a flash-pass item.  The two-launch path keeps one slot per
// item.  The fused launch keeps n_a * kRing slots: item i runs on CTA
// i mod n_a and takes slot i mod (n_a * kRing), last used by the same CTA's
// item i - n_a * kRing.
template <bool FUSED>
__device__ __forceinline__ float *part_ptr(const TcLaunch &L, int item, int h, int row) {
  const int64_t slot = FUSED ? (int64_t)(item % (L.n_a * kRing)) : (int64_t)item;
  return L.partials + ((slot * kPartsPerItem + h) * BM + row) * (D + 4);
}

// Index of an item's (trajectory, layer, KV head) slice in the per-slice counters.
template <class Item>
__device__ __forceinline__ int slice_of(const TcLaunch &L, const Item &it) {
  return (L.slice_off[it.t] + it.li * L.H + it.kvh) * kCounterStride;
}
__device__ __forceinline__ int items_per_slice(const TcLaunch &L, int t) { return L.t[t].nchunk * L.t[t].nrt; }

// Called by all 32 lanes of a warp: waits until *p >= target (an acquire
// load by every lane, so each lane's later reads see the writes released
// with the counter).  Bounded: gives up on the CTA's or the launch's abort
// flag, or after kWait, recording a timeout and raising both flags.
__device__ __forceinline__ bool warp_poll_geq(const uint32_t *p, uint32_t target, volatile int *abort_flag,
                                              WsHeader *hdr) {
  uint64_t t0 = 0;
  for (;;) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    if (__all_sync(0xffffffffu, v >= target)) return true;
    const bool stop = *abort_flag || *reinterpret_cast<volatile int32_t *>(&hdr->abort);
    const uint64_t now = now_ns();
    if (t0 == 0) t0 = now;
    const bool late = now - t0 > kWait;
    if (__any_sync(0xffffffffu, stop || late)) {
      if (late && (threadIdx.x & 31) == 0) {
        *abort_flag = 1;
        atomicExch(&hdr->abort, 1);
        record_error(hdr, COMMITKV_ERR_TIMEOUT, 12);
      }
      return false;
    }
    __nanosleep(512);
  }
}

// Partials of the fused launch are written once and read once soon after:
// kept in L2 over the streaming K and V, dropped first after their read.
__device__ __forceinline__ void st_keep(float *p, float4 v) {
  asm volatile(
      "{\n\t.reg .b64 pol;\n\tcreatepolicy.fractional.L2::evict_last.b64 pol, 1.0;\n\t"
      "st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, pol;\n\t}" ::"l"(p),
      "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
      : "memory");
}
__device__ __forceinline__ float4 ld_once(const float *p) {
  float4 v;
  asm volatile(
      "{\n\t.reg .b64 pol;\n\tcreatepolicy.fractional.L2::evict_first.b64 pol, 1.0;\n\t"
      "ld.global.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], pol;\n\t}"
      : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
      : "l"(p)
      : "memory");
  return v;
}

// Called by all 32 lanes after each wrote its part of a result: one
// release increment of *p for the warp.
__device__ __forceinline__ void signal_add(uint32_t *p, int lane) {
  __threadfence();
  __syncwarp();
  if (lane == 0) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(p) : "memory");
}

template <bool FUSED>
__device__ __forceinline__ void merge_row(const TcLaunch &L, int t, int li, int kvh, int row, int lane);

// ============================================================== pass A
// Two softmax warpgroups take alternate tiles of a chunk (global tile g goes
// to warpgroup g & 1), each with its own S/P buffer, running max, sum and
// output accumulator, so one warpgroup's softmax overlaps the other's MMAs.
// TMEM columns: S/P buffer b at 128 b (after the softmax reads a 32-column
// chunk of S it overwrites the same columns with 16 columns of P_hi and 16
// of P_lo), O_b at 256 + 128 b.  At the end of an item the two warpgroups
// merge their states in the CTA and write one partial.
struct SmemA {
  alignas(1024) uint8_t q[kTileBytes];
  alignas(1024) uint8_t k[NKB][kTileBytes];
  alignas(1024) uint8_t v[NVB][kTileBytes];
  int pos[2][4][BT];  // per softmax warp: positions of the current tile
  float4 pub[BM];     // fused launch: warpgroup 1's (reference max, sum, count, true max) of the item, per row
  uint64_t q_full, q_empty, k_full[NKB], k_empty[NKB], v_full[NVB], v_empty[NVB], s_full[2], s_empty[2], p_full[2],
      pv_done[2], o_full[2], o_empty[2], drain, drain2, pub_full, pub_empty;
  uint32_t tmem;
  int abort_flag;
};

struct ItemA {
  int t, l, kvh, rt, c, li;
};

__device__ __forceinline__ ItemA decode_a(const TcLaunch &L, int item) {
  ItemA it;
  it.t = traj_of(L.item_off_a, L.n_traj, item);
  const TcTraj &tr = L.t[it.t];
  int local = item - L.item_off_a[it.t];
  it.rt = local % tr.nrt;
  local /= tr.nrt;
  it.c = local % tr.nchunk;
  local /= tr.nchunk;
  it.kvh = local % L.H;
  it.li = local / L.H;
  it.l = L.layer_ids[it.li];
  return it;
}

// TMEM column of the 8 packed P columns (hi or lo) of k-step ks inside S/P buffer b.
__device__ __forceinline__ uint32_t p_col(int b, int ks, int lo) {
  return b * BT + 32 * (ks >> 1) + 8 * (ks & 1) + 16 * lo;
}

// Issues S[b] = Q K^T for one tile (8 k-steps over the 128 channels).
__device__ __forceinline__ void issue_qk(uint32_t tm, const uint8_t *q, const uint8_t *k, int b) {
  const uint32_t idesc = idesc_bf16_f32(BM, BT, 0, 0);
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks) mma_bf16(tm + b * BT, desc_kmajor(q, ks), desc_kmajor(k, ks), idesc, ks > 0);
}

// Issues D (+)= P[:, 16 ks .. 16 ks + 15] V[16 ks .. 16 ks + 15, :] with P as
// the (hi, lo) pair in TMEM buffer b; `first` overwrites D.
__device__ __forceinline__ void issue_pv_step(uint32_t tm, uint32_t d_col, const uint8_t *v, int b, int ks,
                                              bool first) {
  const uint32_t idesc = idesc_bf16_f32(BM, D, 0, 1);
  uint64_t bd = desc_v(v, ks);
  mma_bf16_ts(tm + d_col, tm + p_col(b, ks, 0), bd, idesc, first ? 0u : 1u);
  mma_bf16_ts(tm + d_col, tm + p_col(b, ks, 1), bd, idesc, 1u);
}

template <bool FUSED>
__device__ __forceinline__ void flash_body(const TcLaunch &L, WsHeader *hdr, uint8_t *smem_raw, const int cta,
                                           const int ncta) {
  SmemA &sm = *reinterpret_cast<SmemA *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n_items = L.item_off_a[L.n_traj];
  volatile int *abort_flag = &sm.abort_flag;

  if (threadIdx.x == 0) {
    sm.abort_flag = 0;
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, 1);
    for (int s = 0; s < NKB; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
    }
    for (int s = 0; s < NVB; ++s) {
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.s_full[b], 1);
      mbar_init(&sm.s_empty[b], 1);
      mbar_init(&sm.p_full[b], 4);
      mbar_init(&sm.pv_done[b], 1);
      mbar_init(&sm.o_full[b], 1);
      mbar_init(&sm.o_empty[b], 4);
    }
    mbar_init(&sm.drain, 1);
    mbar_init(&sm.drain2, 1);
    mbar_init(&sm.pub_full, 4);   // warpgroup 1's warps: the item's state is published
    mbar_init(&sm.pub_empty, 4);  // warpgroup 0's warps: the publication is consumed
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem;

  // warpgroup 0: TMA producer, P V issuer, Q K^T issuer, one idle warp; 1 and
  // 2: softmax of the even and the odd tiles.  Register budget per thread:
  // 104 + 2 x 200 = the launch's 3 x 168 (the issuers' loops spill below 104;
  // the softmax needs no more than 200).
  if (warp < 4) {
    if (FUSED) regs_dec<48>();
    else regs_dec<104>();  // warp 3 stays idle
    if (warp == 0) {
      // ------------------------------------------------------------ TMA producer
      if (lane == 0) {
        uint64_t pol = policy_evict_normal();
        uint32_t it = 0, n_local = 0, n_k = 0, n_v = 0;  // tiles; Q, K and V copies issued
        bool stop = false;
        for (int item = cta; item < n_items && !stop; item += ncta, ++n_local) {
          if (*abort_flag) break;
          ItemA a = decode_a(L, item);
          const TcTraj &tr = L.t[a.t];
          const TcMaps &mp = L.maps[a.t];
          if (n_local > 0 && !mbar_wait(&sm.q_empty, (n_local - 1) & 1, kWait, abort_flag)) break;
          mbar_expect_tx(&sm.q_full, kTileBytes);
          int qrow = (a.l * L.Hq + a.kvh * L.g) * tr.W + a.rt * BM;
          tma_load_2d(sm.q, &mp.q, 0, qrow, &sm.q_full, pol);
          tma_load_2d(sm.q + kHalf, &mp.q, 64, qrow, &sm.q_full, pol);
          int t0 = a.c * L.chunk_len, t1 = min(tr.S, t0 + L.chunk_len);
          int ntile = (t1 - t0 + BT - 1) / BT;
          // K of tile g once Q K^T of tile g - 3 is done; V once P V of tile g - 2 is
          auto load_k = [&](uint32_t g, int tok) -> bool {
            int s3 = g % NKB;
            if (g >= NKB && !mbar_wait(&sm.k_empty[s3], ((g / NKB) - 1) & 1, kWait, abort_flag)) return false;
            mbar_expect_tx(&sm.k_full[s3], kTileBytes);
            tma4(sm.k[s3], &mp.k, 0, tok, a.kvh, a.l, &sm.k_full[s3], pol);
            tma4(sm.k[s3] + kHalf, &mp.k, 64, tok, a.kvh, a.l, &sm.k_full[s3], pol);
            ++n_k;
            return true;
          };
          auto load_v = [&](uint32_t g, int tok) -> bool {
            int s2 = g % NVB;
            if (g >= NVB && !mbar_wait(&sm.v_empty[s2], ((g / NVB) - 1) & 1, kWait, abort_flag)) return false;
            mbar_expect_tx(&sm.v_full[s2], kTileBytes);
            tma4(sm.v[s2], &mp.v, 0, tok, a.kvh, a.l, &sm.v_full[s2], pol);
            tma4(sm.v[s2] + kHalf, &mp.v, 64, tok, a.kvh, a.l, &sm.v_full[s2], pol);
            ++n_v;
            return true;
          };
          // K runs one tile ahead of V
          if (ntile > 0) stop = !load_k(it, t0);
          for (int j = 0; j < ntile && !stop; ++j) {
            if (j + 1 < ntile && !load_k(it + j + 1, t0 + (j + 1) * BT)) stop = true;
            else if (!load_v(it + j, t0 + j * BT)) stop = true;
          }
          it += ntile;
        }
        if (*abort_flag) {
          // let the copies already issued land before the CTA leaves
          for (uint32_t u = (n_k > NKB ? n_k - NKB : 0); u < n_k; ++u)
            mbar_wait_drain(&sm.k_full[u % NKB], (u / NKB) & 1, kWait);
          for (uint32_t u = (n_v > NVB ? n_v - NVB : 0); u < n_v; ++u)
            mbar_wait_drain(&sm.v_full[u % NVB], (u / NVB) & 1, kWait);
          if (n_local > 0) mbar_wait_drain(&sm.q_full, (n_local - 1) & 1, kWait);
        }
      }
  } else if (warp == 1) {
    // ------------------------------------------------------------ P V issuer
    if (lane == 0) {
      uint32_t it = 0;
      int uses0 = 0, uses1 = 0;  // items in which O_0 / O_1 have been filled so far
      bool ok = true;
      for (int item = cta; item < n_items && ok; item += ncta) {
        ItemA a = decode_a(L, item);
        const TcTraj &tr = L.t[a.t];
        int t0 = a.c * L.chunk_len, t1 = min(tr.S, t0 + L.chunk_len);
        int ntile = (t1 - t0 + BT - 1) / BT;
        for (int j = 0; j < ntile && ok; ++j) {
          uint32_t g = it + j;
          int s2 = g % NVB, b = g & 1;
          const bool first = j < 2, last = j + 2 >= ntile;  // of warpgroup b in this item
          // O_b of the previous item must have been read out before P V overwrites it
          const int ub = b ? uses1 : uses0;
          if (first && ub > 0 && !mbar_wait(&sm.o_empty[b], (ub - 1) & 1, kWait, abort_flag)) {
            ok = false;
            break;
          }
          if (!mbar_wait(&sm.p_full[b], (g >> 1) & 1, kWait, abort_flag) ||
              !mbar_wait(&sm.v_full[s2], (g / NVB) & 1, kWait, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < BT / 16; ++ks) issue_pv_step(tm, 2 * BT + b * D, sm.v[s2], b, ks, first && ks == 0);
          mma_commit(&sm.s_empty[b]);
          mma_commit(&sm.v_empty[s2]);
          mma_commit(&sm.pv_done[b]);
          if (last) {
            mma_commit(&sm.o_full[b]);
            if (b) ++uses1;
            else ++uses0;
          }
        }
        it += ntile;
      }
      if (*abort_flag) {
        mma_commit(&sm.drain);  // every MMA issued by this thread has completed
        mbar_wait_drain(&sm.drain, 0, kWait);
      }
    }
    } else if (warp == 2) {
      // ------------------------------------------------------------ Q K^T issuer
      if (lane == 0) {
        uint32_t it = 0, n_local = 0;
        bool ok = true;
        for (int item = cta; item < n_items && ok; item += ncta, ++n_local) {
          ItemA a = decode_a(L, item);
          const TcTraj &tr = L.t[a.t];
          int t0 = a.c * L.chunk_len, t1 = min(tr.S, t0 + L.chunk_len);
          int ntile = (t1 - t0 + BT - 1) / BT;
          if (!mbar_wait(&sm.q_full, n_local & 1, kWait, abort_flag)) break;
          tc_fence_after();
          for (int j = 0; j < ntile && ok; ++j) {
            uint32_t g = it + j;
            int s3 = g % NKB, b = g & 1;
            if (!mbar_wait(&sm.k_full[s3], (g / NKB) & 1, kWait, abort_flag) ||
                (g >= 2 && !mbar_wait(&sm.s_empty[b], ((g >> 1) - 1) & 1, kWait, abort_flag))) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_qk(tm, sm.q, sm.k[s3], b);
            mma_commit(&sm.s_full[b]);
            mma_commit(&sm.k_empty[s3]);
            if (j + 1 == ntile) mma_commit(&sm.q_empty);  // every Q K^T of this item is issued
          }
          it += ntile;
        }
        if (*abort_flag) {
          mma_commit(&sm.drain2);  // every MMA issued by this thread has completed
          mbar_wait_drain(&sm.drain2, 0, kWait);
        }
      }
    }
  } else if (warp < 12) {
    // ------------------------------------------------------------ softmax (warps 4..11)
    if (FUSED) regs_inc<208>();
    else regs_inc<200>();
    const int hb = (warp - 4) >> 2;   // this warpgroup's tiles: g & 1 == hb
    const int wq = warp & 3;          // TMEM lane quarter of this warp
    const int row = wq * 32 + lane;   // probe row within the tile
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    const uint32_t o_col = 2 * BT + hb * D;
    int *posw = sm.pos[hb][wq];
    uint32_t it = 0;
    int uses = 0;  // items in which this warpgroup filled O_hb
    uint32_t n_it = 0;  // items of this CTA seen so far (fused launch)
    bool ok = true;
    for (int item = cta; item < n_items && ok; item += ncta) {
      ItemA a = decode_a(L, item);
      const TcTraj &tr = L.t[a.t];
      int rows = L.g * tr.W;
      int grow = a.rt * BM + row;  // row within the (layer, KV head) slice
      bool valid_row = grow < rows;
      int qp = valid_row ? tr.qpos[grow % tr.W] : -0x7fffffff;
      const int vis_all = tr.prep->vis_all;
      int t0 = a.c * L.chunk_len, t1 = min(tr.S, t0 + L.chunk_len);
      int ntile = (t1 - t0 + BT - 1) / BT;
      const int j0 = (hb - (int)it) & 1;  // first tile of this warpgroup in the item
      float *dst = part_ptr<FUSED>(L, item, hb, row);
      float m_used = -INFINITY, m_true = -INFINITY, lsum = 0.0f;
      int nvis = 0;
      for (int j = j0; j < ntile && ok; j += 2) {
        uint32_t g = it + j;
        const int b = hb;
        int tok0 = t0 + j * BT, nt = min(BT, t1 - tok0);
        // tiles inside the prefix every probe row sees need no position test
        const bool full = tok0 + nt <= vis_all;
        if (!full) {  // each warp keeps its own copy: no cross-warp barrier
          __syncwarp();
#pragma unroll
          for (int i = lane; i < BT; i += 32) posw[i] = i < nt ? tr.pos[tok0 + i] : 0x7fffffff;
          __syncwarp();
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[b], (g >> 1) & 1, kWait, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        // visibility of column i: inside the tile and, outside the prefix every
        // probe row sees, at or before the row's query position
        const bool simple = full && nt == BT && valid_row;
        // sweep 1: row max over the tile, 32 columns at a time
        float mx[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) mx[k] = -INFINITY;
        int cnt = simple ? BT : 0;
#pragma unroll 1
        for (int c0 = 0; c0 < BT; c0 += 32) {
          float x[32];
          tmem_ld32f(tm + lane_base + b * BT + c0, x);
          tmem_wait_ld();
          if (!simple) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              bool vis = valid_row && c0 + i < nt && (full || posw[c0 + i] <= qp);
              x[i] = vis ? x[i] : -INFINITY;
              cnt += vis;
            }
          }
#pragma unroll
          for (int i = 0; i < 32; i += 8)
#pragma unroll
            for (int k = 0; k < 8; ++k) mx[k] = fmaxf(mx[k], x[i + k]);
        }
        float smax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
        float mt = smax == -INFINITY ? smax : smax * L.scale_log2;
        nvis += cnt;
        m_true = fmaxf(m_true, mt);
        float m_new = fmaxf(m_used, mt);
        bool rescale = m_new > m_used + kLazy;  // false while both are -inf
        float alpha = (rescale && m_used != -INFINITY) ? exp2f(m_used - m_new) : 0.0f;
        if (rescale) m_used = m_new;
        if (j > j0) {
          // P V of this warpgroup's previous tile done: O_hb is stable
          if (!__all_sync(0xffffffffu, mbar_wait(&sm.pv_done[b], ((g >> 1) - 1) & 1, kWait, abort_flag))) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (__any_sync(0xffffffffu, rescale)) {
            float f = rescale ? alpha : 1.0f;
#pragma unroll
            for (int c0 = 0; c0 < D; c0 += 32) {
              uint32_t r[32];
              tmem_ld32(tm + lane_base + o_col + c0, r);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * f);
              tmem_st32(tm + lane_base + o_col + c0, r);
            }
            tmem_wait_st();
          }
        }
        if (rescale) lsum *= alpha;
        const float neg_m = m_used == -INFINITY ? 0.0f : -m_used;
        // sweep 2: p = 2^(s c - m) on the visible columns (2^-inf = 0), the row
        // sum, and P as the (hi, lo) bf16 pair over the S columns just read
        float pacc[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) pacc[k] = 0.0f;
#pragma unroll 1
        for (int c0 = 0; c0 < BT; c0 += 32) {
          float x[32];
          tmem_ld32f(tm + lane_base + b * BT + c0, x);
          tmem_wait_ld();
          if (!simple) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              bool vis = valid_row && c0 + i < nt && (full || posw[c0 + i] <= qp);
              x[i] = vis ? x[i] : -INFINITY;
            }
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) x[i] = fast_exp2(fmaf(x[i], L.scale_log2, neg_m));
#pragma unroll
          for (int i = 0; i < 32; i += 8)
#pragma unroll
            for (int k = 0; k < 8; ++k) pacc[k] += x[i + k];
          uint32_t pk[32];
          split_pack32(x, pk);
          tmem_st32(tm + lane_base + b * BT + c0, pk);
        }
        float ps = ((pacc[0] + pacc[1]) + (pacc[2] + pacc[3])) + ((pacc[4] + pacc[5]) + (pacc[6] + pacc[7]));
        tmem_wait_st();
        lsum += ps;
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.p_full[b]);
      }
      if (!ok) break;
      {
        // One partial per item: warpgroup 1 publishes its (reference max,
        // sum, count, true max) and leaves its O in tensor memory; warpgroup
        // 0 rescales both outputs to the larger reference max, writes the
        // partial and hands both O accumulators back to the P V issuer.
        const bool mine = j0 < ntile;  // this warpgroup filled its O in this item
        if (hb == 1) {
          if (n_it > 0 && !__all_sync(0xffffffffu, mbar_wait(&sm.pub_empty, (n_it - 1) & 1, kWait, abort_flag))) {
            ok = false;
            break;
          }
          if (mine && !__all_sync(0xffffffffu, mbar_wait(&sm.o_full[1], uses & 1, kWait, abort_flag))) {
            ok = false;
            break;
          }
          sm.pub[row] = make_float4(mine ? m_used : -INFINITY, lsum, (float)nvis, m_true);
          if (mine) ++uses;
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.pub_full);
        } else {
          if (FUSED && item >= L.n_a * kRing) {
            // the partial slot was last used by this CTA's item kRing items
            // back: its slice must be merged before the slot is overwritten
            const ItemA pa = decode_a(L, item - L.n_a * kRing);
            if (!warp_poll_geq(&L.merged[slice_of(L, pa)], 4u * items_per_slice(L, pa.t), abort_flag, hdr)) {
              ok = false;
              break;
            }
          }
          if ((mine && !__all_sync(0xffffffffu, mbar_wait(&sm.o_full[0], uses & 1, kWait, abort_flag))) ||
              !__all_sync(0xffffffffu, mbar_wait(&sm.pub_full, n_it & 1, kWait, abort_flag))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float4 o1 = sm.pub[row];
          const bool mine1 = (int)((1u - it) & 1u) < ntile;  // warpgroup 1 filled its O in this item
          const bool theirs = mine1 && o1.x != -INFINITY;
          const float m0 = mine ? m_used : -INFINITY;
          const float mr = fmaxf(m0, theirs ? o1.x : -INFINITY);
          const float f0 = m0 == -INFINITY ? 0.0f : exp2f(m0 - mr);
          const float f1 = theirs ? exp2f(o1.x - mr) : 0.0f;
#pragma unroll 1
          for (int c0 = 0; c0 < D; c0 += 32) {
            float x0[32], x1[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) x0[i] = x1[i] = 0.0f;
            if (mine) tmem_ld32f(tm + lane_base + 2 * BT + c0, x0);
            if (mine1) tmem_ld32f(tm + lane_base + 2 * BT + D + c0, x1);
            tmem_wait_ld();
            if (valid_row) {
#pragma unroll
              for (int i = 0; i < 32; i += 4) {
                const float4 v = make_float4(fmaf(x0[i], f0, theirs ? x1[i] * f1 : 0.0f),
                                             fmaf(x0[i + 1], f0, theirs ? x1[i + 1] * f1 : 0.0f),
                                             fmaf(x0[i + 2], f0, theirs ? x1[i + 2] * f1 : 0.0f),
                                             fmaf(x0[i + 3], f0, theirs ? x1[i + 3] * f1 : 0.0f));
                // the fused launch's merge reads the partial soon: keep it in L2
                if (FUSED) st_keep(dst + 4 + c0 + i, v);
                else *reinterpret_cast<float4 *>(dst + 4 + c0 + i) = v;
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (mine) mbar_arrive(&sm.o_empty[0]);
            if (mine1) mbar_arrive(&sm.o_empty[1]);
            mbar_arrive(&sm.pub_empty);
          }
          if (mine) ++uses;
          // (reference max of l and O, sum, visible count, true max)
          if (valid_row) {
            const float4 hd = make_float4(mr, fmaf(lsum, f0, o1.y * f1), (float)nvis + o1.z, fmaxf(m_true, o1.w));
            if (FUSED) st_keep(dst, hd);
            else *reinterpret_cast<float4 *>(dst) = hd;
          }
          if (FUSED) signal_add(&L.a_done[slice_of(L, a)], lane);  // this warp's rows of the partial are written
        }
        ++n_it;
        it += ntile;
      }
    }
  } else if (FUSED) {
    // ------------------------------------------------------------ merge (warps 12..15, fused launch only)
    // For each item of this CTA, once every item of its slice has written
    // its partials, the four warps merge this item's share of the slice's
    // probe rows into the row statistics (m, l, n, o); the page-pass CTAs
    // wait for all shares of a slice.  No tensor memory, no TMA.
    regs_dec<48>();
    const int w = warp - 12;
    for (int item = cta; item < n_items; item += ncta) {
      const ItemA a = decode_a(L, item);
      const TcTraj &tr = L.t[a.t];
      const int s = slice_of(L, a), nis = items_per_slice(L, a.t);
      if (!warp_poll_geq(&L.a_done[s], 4u * nis, abort_flag, hdr)) break;
      const int rows = L.g * tr.W, jin = a.c * tr.nrt + a.rt;
      const int r0 = (int)((int64_t)jin * rows / nis), r1 = (int)((int64_t)(jin + 1) * rows / nis);
      for (int row = r0 + w; row < r1; row += 4) merge_row<FUSED>(L, a.t, a.li, a.kvh, row, lane);
      signal_add(&L.merged[s], lane);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tm, 512);
  if (threadIdx.x == 0 && sm.abort_flag) {
    if (FUSED) atomicExch(&hdr->abort, 1);
    record_error(hdr, COMMITKV_ERR_TIMEOUT, 10);
  }
}

__global__ void __launch_bounds__(384, 1) pass_a_tc(const __grid_constant__ TcLaunch L, WsHeader *hdr) {
  extern __shared__ uint8_t smem_raw[];
  flash_body<false>(L, hdr, smem_raw, blockIdx.x, gridDim.x);
}


// ============================================================== combine
// Merges the 2 x nchunk partials of one probe row of a (trajectory, layer,
// KV head) slice into its row stats (m, l, n, o): one warp, four channels
// per lane.
template <bool FUSED>
__device__ __forceinline__ void merge_row(const TcLaunch &L, int t, int li, int kvh, int row, int lane) {
  const TcTraj &tr = L.t[t];
  const int l = L.layer_ids[li];
  const int rt = row / BM, rl = row % BM;
  // partial k = chunk k (one per item: the two softmax warpgroups' states
  // are merged in the CTA)
  auto part = [&](int k) {
    const int item = L.item_off_a[t] + ((li * L.H + kvh) * tr.nchunk + k) * tr.nrt + rt;
    return part_ptr<FUSED>(L, item, 0, rl);
  };
  const int nparts = tr.nchunk;  // at most 32 (checked on the host)
  // headers, one partial per lane: (reference max, sum, visible count, true max)
  const float4 h0 = lane < nparts ? ld_once(part(lane)) : make_float4(-INFINITY, 0.f, 0.f, -INFINITY);
  const float4 h1 = lane + 32 < nparts ? ld_once(part(lane + 32)) : make_float4(-INFINITY, 0.f, 0.f, -INFINITY);
  // the first kBatch partials' outputs, four channels per lane, loaded
  // before the weights are known (the loads depend on nothing)
  constexpr int kBatch = FUSED ? 2 : 8;  // the fused launch's merge warps run on 48 registers
  float4 vb[kBatch];
#pragma unroll
  for (int u = 0; u < kBatch; ++u) vb[u] = u < nparts ? ld_once(part(u) + 4 + lane * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float m = warp_max(fmaxf(h0.w, h1.w));  // true row max over the partials (base 2)
  // weight of each partial; a partial that saw nothing (reference -inf) has
  // weight 0 and an unwritten output
  const float a0 = h0.x == -INFINITY ? 0.0f : exp2f(h0.x - m);
  const float a1 = h1.x == -INFINITY ? 0.0f : exp2f(h1.x - m);
  const float lsum = warp_sum(fmaf(h0.y, a0, h1.y * a1));
  const float n = warp_sum(h0.z + h1.z);
  float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
  // outputs, partials in order, in batches whose loads are issued
  // together
  for (int k0 = 0; k0 < nparts; k0 += kBatch) {
    if (k0 > 0) {
#pragma unroll
      for (int u = 0; u < kBatch; ++u)
        vb[u] = k0 + u < nparts ? ld_once(part(k0 + u) + 4 + lane * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int k = k0 + u;
      const float a = __shfl_sync(0xffffffffu, k < 32 ? a0 : a1, k & 31);
      if (k >= nparts) break;
      float4 v = vb[u];
      if (a == 0.0f) v = make_float4(0.f, 0.f, 0.f, 0.f);
      o.x = fmaf(v.x, a, o.x);
      o.y = fmaf(v.y, a, o.y);
      o.z = fmaf(v.z, a, o.z);
      o.w = fmaf(v.w, a, o.w);
    }
  }
  const float inv = lsum > 0.0f ? 1.0f / lsum : 0.0f;
  const int h = kvh * L.g + row / tr.W, w = row % tr.W;
  float *dst = tr.stats + (((int64_t)l * L.Hq + h) * tr.W + w) * (D + 4);
  if (lane == 0)
    *reinterpret_cast<float4 *>(dst) = make_float4(m == -INFINITY ? m : m * 0.69314718055994531f, lsum, n, 0.0f);
  *reinterpret_cast<float4 *>(dst + 4 + lane * 4) = make_float4(o.x * inv, o.y * inv, o.z * inv, o.w * inv);
}

// One warp per probe row of the selected layers (the two-launch path).
__global__ void __launch_bounds__(256) combine_tc(const __grid_constant__ TcLaunch L) {
  const int gw = (blockIdx.x * 256 + threadIdx.x) / 32, lane = threadIdx.x % 32;
  if (gw >= L.row_off[L.n_traj]) return;
  const int t = traj_of(L.row_off, L.n_traj, gw);
  const TcTraj &tr = L.t[t];
  int local = gw - L.row_off[t];
  const int rows = L.g * tr.W;
  const int row = local % rows;
  local /= rows;
  merge_row<false>(L, t, local / L.H, local % L.H, row, lane);
}

// ============================================================== prep
// Per trajectory, once per call:
//   slot_off[E] = sum over F < E of ceil(len_F / 16), slot_off[P] = total
//   (a page that fails the table checks gets no slot and an error is recorded);
//   slot_tab[slot] = {first token, valid tokens, page, first/last flags and
//   the page's rank among the pages with slots} for every 16-token slot;
//   the pass-B work items: item k takes the pages whose first slot lies in
//   [k * slots_per_item, (k + 1) * slots_per_item);
//   vis_all = number of leading resident tokens visible to every probe row
//   (positions increase, so this is a prefix); nvis_w[w] = number of resident
//   tokens visible to window position w.
__global__ void __launch_bounds__(1024) prep_kernel(const __grid_constant__ TcLaunch L, WsHeader *hdr) {
  const TcTraj &tr = L.t[blockIdx.x];
  int lane = threadIdx.x % 32, wid = threadIdx.x / 32;
  // one scan gives both the slot offsets (low 32 bits) and the rank of each
  // page among the pages that have slots (high 32 bits)
  __shared__ unsigned long long s_w64[32];
  __shared__ unsigned long long s_b64;
  if (threadIdx.x == 0) s_b64 = 0ull;
  __syncthreads();
  for (int c0 = 0; c0 < tr.P; c0 += 1024) {
    int E = c0 + threadIdx.x;
    int ns = 0, ps = 0, pl = 0;
    if (E < tr.P) {
      ps = tr.ps[E];
      pl = tr.pl[E];
      bool bad = pl < 0 || ps < 0 || ps > tr.S - pl || (E > 0 && ps < tr.ps[E - 1] + tr.pl[E - 1]);
      if (bad) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, E);
      ns = bad ? 0 : (pl + SLOT - 1) / SLOT;
    }
    const unsigned long long v = ((unsigned long long)(ns > 0) << 32) | (unsigned)ns;
    unsigned long long x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_w64[wid] = x;
    __syncthreads();
    if (wid == 0) {
      unsigned long long w = s_w64[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        unsigned long long y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      s_w64[lane] = w;
    }
    __syncthreads();
    const unsigned long long excl = s_b64 + (wid ? s_w64[wid - 1] : 0ull) + x - v;
    if (E < tr.P) {
      const int off = (int)(excl & 0xffffffffull), rank = (int)(excl >> 32);
      tr.slot_off[E] = off;
      for (int sub = 0; sub < ns; ++sub)
        tr.slot_tab[off + sub] = make_int4(ps + sub * SLOT, min(SLOT, pl - sub * SLOT), E,
                                           (sub == 0 ? 1 : 0) | (sub + 1 == ns ? 2 : 0) | (rank << 2));
    }
    __syncthreads();
    if (threadIdx.x == 0) s_b64 += s_w64[31];
    __syncthreads();
  }
  if (threadIdx.x == 0) tr.slot_off[tr.P] = (int)(s_b64 & 0xffffffffull);
  __syncthreads();
  for (int k = threadIdx.x; k < tr.nbitem; k += 1024) {
    int lo = k * L.slots_per_item, hi = lo + L.slots_per_item;
    int a = 0, b = tr.P;
    while (a < b) {
      int mid = (a + b) >> 1;
      if (tr.slot_off[mid] < lo) a = mid + 1;
      else b = mid;
    }
    int E0 = a;
    b = tr.P;
    while (a < b) {
      int mid = (a + b) >> 1;
      if (tr.slot_off[mid] < hi) a = mid + 1;
      else b = mid;
    }
    int E1 = a;
    int slot0 = E0 < tr.P ? tr.slot_off[E0] : 0;
    int nslot = E1 > E0 ? tr.slot_off[E1] - slot0 : 0;
    int npages = 0;
    for (int E = E0; E < E1; ++E) npages += tr.slot_off[E + 1] > tr.slot_off[E];
    tr.items[2 * k] = make_int4(E0, E1, slot0, nslot);
    tr.items[2 * k + 1] = make_int4(npages, 0, 0, 0);
  }
  for (int w = threadIdx.x; w < tr.W; w += blockDim.x) {
    const int qp = tr.qpos[w];
    int a = 0, b = tr.S;
    while (a < b) {
      int mid = (a + b) >> 1;
      if (tr.pos[mid] <= qp) a = mid + 1;
      else b = mid;
    }
    tr.nvis_w[w] = a;
  }
  if (threadIdx.x == 0) {
    int qmin = 0x7fffffff;
    for (int w = 0; w < tr.W; ++w) qmin = min(qmin, tr.qpos[w]);
    int a = 0, b = tr.S;  // first token with pos > qmin
    while (a < b) {
      int mid = (a + b) >> 1;
      if (tr.pos[mid] <= qmin) a = mid + 1;
      else b = mid;
    }
    tr.prep->vis_all = a;
  }
}

// ============================================================== pass B
// TMEM columns: S/P buffers at 0 and 128 (as in pass A), page accumulators
// U[0] at 256 and U[1] at 384.
struct SlotMeta {
  int tok0;   // first resident index of the slot
  int nv;     // valid tokens in the slot (0 for an empty slot)
  int po;     // page ordinal within the CTA's page stream (-1: empty slot)
  int flags;  // bit 0: first slot of its page, bit 1: last slot of its page
};

struct SmemB {
  alignas(1024) uint8_t q[kTileBytes];
  alignas(1024) uint8_t k[NKB][kTileBytes];
  alignas(1024) uint8_t v[NVB][kTileBytes];
  SlotMeta meta[NKB][SLOTS];
  int page_of[NKB][SLOTS];  // page id of each slot
  uint32_t tile_bytes[NKB]; // bytes of the tile's K (and V) copies
  int tile_full[NKB];       // every slot of the tile lies in the prefix all probe rows see
  int pos[4][BT];           // per softmax warp: positions of the current tile
  float fifo_s[NFIFO][BM];  // per page: S_E of every row
  int fifo_n[NFIFO][BM];    // per page: visible count of every row
  int fifo_page[NFIFO];
  uint64_t q_full, q_empty, k_full[NKB], k_empty[NKB], meta_empty[NKB], v_full[NVB], v_empty[NVB], s_full[2],
      s_empty[2], p_full[2], acc_full[2], acc_empty[2], fifo_full[NFIFO], fifo_empty[NFIFO], drain[2], drain2;
  uint32_t tmem;
  int abort_flag;
};

struct ItemB {
  int t, l, kvh, rt, k, li;
  int E0, E1;        // pages [E0, E1)
  int slot0, nslot;  // slots of those pages
};

__device__ __forceinline__ ItemB decode_b(const TcLaunch &L, int item) {
  ItemB b;
  b.t = traj_of(L.item_off_b, L.n_traj, item);
  const TcTraj &tr = L.t[b.t];
  int local = item - L.item_off_b[b.t];
  b.rt = local % tr.nrt;
  local /= tr.nrt;
  b.k = local % tr.nbitem;
  local /= tr.nbitem;
  b.kvh = local % L.H;
  b.li = local / L.H;
  b.l = L.layer_ids[b.li];
  int4 e = tr.items[2 * b.k];
  b.E0 = e.x;
  b.E1 = e.y;
  b.slot0 = e.z;
  b.nslot = e.w;
  return b;
}

template <bool FUSED>
__device__ __forceinline__ void page_body(const TcLaunch &L, WsHeader *hdr, uint8_t *smem_raw, const int cta,
                                          const int ncta) {
  SmemB &sm = *reinterpret_cast<SmemB *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n_items = L.item_off_b[L.n_traj];
  volatile int *abort_flag = &sm.abort_flag;

  if (threadIdx.x == 0) {
    sm.abort_flag = 0;
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, 1);
    for (int s = 0; s < NKB; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
      mbar_init(&sm.meta_empty[s], 6);  // four softmax warps and the two P V threads
    }
    for (int s = 0; s < NVB; ++s) {
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.v_empty[s], 2);  // both P V threads
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.s_full[b], 1);
      mbar_init(&sm.s_empty[b], 2);  // both P V threads
      mbar_init(&sm.acc_full[b], 1);
      mbar_init(&sm.acc_empty[b], 4);  // the epilogue warpgroup of that page parity
    }
    // one per S/P buffer: the softmax can finish tile g + 1 before the P V
    // thread has seen tile g, but not tile g + 2, so a parity wait on a
    // per-buffer barrier cannot miss a phase
    mbar_init(&sm.p_full[0], 4);
    mbar_init(&sm.p_full[1], 4);
    for (int f = 0; f < NFIFO; ++f) {
      mbar_init(&sm.fifo_full[f], 4);
      mbar_init(&sm.fifo_empty[f], 4);
    }
    mbar_init(&sm.drain[0], 1);
    mbar_init(&sm.drain[1], 1);
    mbar_init(&sm.drain2, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem;

  // warpgroup 0: TMA producer, two P V issuers (warps 1 and 3), Q K^T issuer; 1: softmax;
  // 2 and 3: epilogue.  Each branch first sets its warpgroup's register
  // budget: 64 + 112 + 2 x 168 per thread = the launch's 4 x 128 (a budget
  // below 128 is set with a decrease, above it with an increase).
  if (warp < 4) {
    regs_dec<64>();
    if (warp == 0) {
      // ------------------------------------------------------------ TMA producer
      // The whole warp works each tile: lanes 0..7 take one 16-token slot each
      // from the slot table, write the tile's slot table to shared memory and
      // issue the copies of the runs of slots that start at them.
      uint64_t pol = policy_evict_first();
      uint32_t it = 0, n_local = 0, n_k = 0, n_v = 0;  // tiles; Q, K and V copies issued
      int po_base = 0;  // page ordinal of the item's first page
      bool stop = false;
      for (int item = cta; item < n_items && !stop; item += ncta) {
        if (*abort_flag) break;
        ItemB bi = decode_b(L, item);
        if (bi.nslot == 0) continue;
        const TcTraj &tr = L.t[bi.t];
        const TcMaps &mp = L.maps[bi.t];
        const int4 *stab = tr.slot_tab + bi.slot0;
        const int rank0 = stab[0].w >> 2;  // slotted-page rank of the item's first page
        const int vis_all = tr.prep->vis_all;
        if (n_local > 0 && !__all_sync(0xffffffffu, mbar_wait(&sm.q_empty, (n_local - 1) & 1, kWait, abort_flag))) {
          stop = true;
          break;
        }
        if (lane == 0) {
          mbar_expect_tx(&sm.q_full, kTileBytes);
          int qrow = (bi.l * L.Hq + bi.kvh * L.g) * tr.W + bi.rt * BM;
          tma_load_2d(sm.q, &mp.q, 0, qrow, &sm.q_full, pol);
          tma_load_2d(sm.q + kHalf, &mp.q, 64, qrow, &sm.q_full, pol);
        }
        ++n_local;
        // Copies of the runs of slots whose rows are contiguous in memory (full
        // slots of one event): a lane that starts a run issues its boxes of 16,
        // 32, 64 or 128 rows.  Called by the whole warp; lanes 0..7 carry a slot.
        auto issue_runs = [&](int tok0, int nv, bool valid, uint8_t *dst, const CUtensorMap *big,
                              const CUtensorMap *small, uint64_t *bar) {
          unsigned vmask = __ballot_sync(0xffffffffu, valid);
          int ptok = __shfl_up_sync(0xffffffffu, tok0, 1), pnv = __shfl_up_sync(0xffffffffu, nv, 1);
          bool pvalid = lane > 0 && ((vmask >> (lane - 1)) & 1u);
          bool start = valid && (!pvalid || pnv != SLOT || ptok + SLOT != tok0);
          unsigned smask = __ballot_sync(0xffffffffu, start);
          if (start) {
            unsigned ends = (smask | ~vmask) & ~((2u << lane) - 1u);  // run boundaries after this lane
            int run = (__ffs(ends) - 1) - lane;                        // lanes >= 8 are never valid
            int done = 0;
            while (done < run) {
              int rem = run - done;
              int lg = rem >= 8 ? 3 : rem >= 4 ? 2 : rem >= 2 ? 1 : 0;
              if (lg == 3 && (lane + done) != 0) lg = 2;  // a 128-row box covers the whole tile
              int tok = tok0 + done * SLOT;
              uint8_t *d = dst + (lane + done) * SLOT * 128;
              const CUtensorMap *m = lg == 3 ? big : small + lg;
              tma4(d, m, 0, tok, bi.kvh, bi.l, bar, pol);
              tma4(d + kHalf, m, 64, tok, bi.kvh, bi.l, bar, pol);
              done += 1 << lg;
            }
          }
        };
        // K of tile g (and its slot table) once Q K^T of tile g - 3 is done and
        // its slot table released
        auto load_k = [&](uint32_t g, int j) -> bool {
          int s3 = g % NKB;
          bool w_ok = g < NKB || (mbar_wait(&sm.k_empty[s3], ((g / NKB) - 1) & 1, kWait, abort_flag) &&
                                  mbar_wait(&sm.meta_empty[s3], ((g / NKB) - 1) & 1, kWait, abort_flag));
          if (!__all_sync(0xffffffffu, w_ok)) return false;
          int sl = j * SLOTS + lane;
          bool valid = lane < SLOTS && sl < bi.nslot;
          int4 rec = valid ? stab[sl] : make_int4(0, 0, -1, 0);
          SlotMeta mt;
          mt.tok0 = rec.x;
          mt.nv = valid ? rec.y : 0;
          mt.po = valid ? po_base + (rec.w >> 2) - rank0 : -1;
          mt.flags = valid ? rec.w & 3 : 0;
          if (lane < SLOTS) {
            sm.meta[s3][lane] = mt;
            sm.page_of[s3][lane] = rec.z;
          }
          const bool tfull = __all_sync(0xffffffffu, !valid || rec.x + rec.y <= vis_all);
          const uint32_t bytes = __popc(__ballot_sync(0xffffffffu, valid)) * 2u * SLOT * 128u;
          __syncwarp();  // the slot table is written before the arrival that publishes it
          if (lane == 0) {
            sm.tile_bytes[s3] = bytes;
            sm.tile_full[s3] = tfull;
            mbar_expect_tx(&sm.k_full[s3], bytes);
          }
          __syncwarp();
          issue_runs(mt.tok0, mt.nv, valid, sm.k[s3], &mp.k, mp.kb, &sm.k_full[s3]);
          ++n_k;
          return true;
        };
        // V of tile g once P V of tile g - 2 is done
        auto load_v = [&](uint32_t g) -> bool {
          int s3 = g % NKB, s2 = g % NVB;
          bool w_ok = g < NVB || mbar_wait(&sm.v_empty[s2], ((g / NVB) - 1) & 1, kWait, abort_flag);
          if (!__all_sync(0xffffffffu, w_ok)) return false;
          SlotMeta mt = sm.meta[s3][lane < SLOTS ? lane : 0];
          bool valid = lane < SLOTS && mt.po >= 0;
          if (lane == 0) mbar_expect_tx(&sm.v_full[s2], sm.tile_bytes[s3]);
          __syncwarp();
          issue_runs(mt.tok0, mt.nv, valid, sm.v[s2], &mp.v, mp.vb, &sm.v_full[s2]);
          ++n_v;
          return true;
        };
        // K runs one tile ahead of V
        int ntile = (bi.nslot + SLOTS - 1) / SLOTS;
        stop = !load_k(it, 0);
        for (int j = 0; j < ntile && !stop; ++j) {
          if (j + 1 < ntile && !load_k(it + j + 1, j + 1)) stop = true;
          else if (!load_v(it + j)) stop = true;
        }
        it += ntile;
        po_base += tr.items[2 * bi.k + 1].x;
      }
      if (lane == 0 && *abort_flag) {
        // let the copies already issued land before the CTA leaves
        for (uint32_t u = (n_k > NKB ? n_k - NKB : 0); u < n_k; ++u)
          mbar_wait_drain(&sm.k_full[u % NKB], (u / NKB) & 1, kWait);
        for (uint32_t u = (n_v > NVB ? n_v - NVB : 0); u < n_v; ++u)
          mbar_wait_drain(&sm.v_full[u % NVB], (u / NVB) & 1, kWait);
        if (n_local > 0) mbar_wait_drain(&sm.q_full, (n_local - 1) & 1, kWait);
      }
    } else if (warp == 1 || warp == 3) {
      // ------------------------------------------------------------ P V issuers
      // Two issuing threads, one per page accumulator: warp 1 the even page
      // ordinals (U[0]), warp 3 the odd ones (U[1]).  Both release the S/P
      // buffer, the V stage and the slot table of every tile.
      const int par = warp == 1 ? 0 : 1;
      if (lane == 0) {
        uint32_t it = 0;
        bool ok = true;
        for (int item = cta; item < n_items && ok; item += ncta) {
          ItemB bi = decode_b(L, item);
          if (bi.nslot == 0) continue;
          int ntile = (bi.nslot + SLOTS - 1) / SLOTS;
          for (int j = 0; j < ntile && ok; ++j) {
            uint32_t g = it + j;
            int s3 = g % NKB, s2 = g % NVB, b = g & 1;
            if (!mbar_wait(&sm.p_full[b], (g >> 1) & 1, kWait, abort_flag) ||
                !mbar_wait(&sm.v_full[s2], (g / NVB) & 1, kWait, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll 1
            for (int q = 0; q < SLOTS && ok; ++q) {
              SlotMeta mt = sm.meta[s3][q];
              if (mt.po < 0 || (mt.po & 1) != par) continue;
              const int a = par;
              if ((mt.flags & 1) && mt.po >= 2) {
                if (!mbar_wait(&sm.acc_empty[a], ((mt.po >> 1) - 1) & 1, kWait, abort_flag)) {
                  ok = false;
                  break;
                }
                tc_fence_after();
              }
              issue_pv_step(tm, 2 * BT + a * D, sm.v[s2], b, q, (mt.flags & 1) != 0);
              if (mt.flags & 2) mma_commit(&sm.acc_full[a]);
            }
            mma_commit(&sm.s_empty[b]);
            mma_commit(&sm.v_empty[s2]);
            mbar_arrive(&sm.meta_empty[s3]);  // done with the slot table
          }
          it += ntile;
        }
        if (*abort_flag) {
          mma_commit(&sm.drain[par]);  // every MMA issued by this thread has completed
          mbar_wait_drain(&sm.drain[par], 0, kWait);
        }
      }
    } else if (warp == 2) {
      // ------------------------------------------------------------ Q K^T issuer
      // A second issuing thread: S = Q K^T of tile g needs only its K copy and
      // the S/P buffer that P V of tile g - 2 has finished reading.
      if (lane == 0) {
        uint32_t it = 0, n_local = 0;
        bool ok = true;
        for (int item = cta; item < n_items && ok; item += ncta) {
          ItemB bi = decode_b(L, item);
          if (bi.nslot == 0) continue;
          int ntile = (bi.nslot + SLOTS - 1) / SLOTS;
          if (!mbar_wait(&sm.q_full, n_local & 1, kWait, abort_flag)) break;
          ++n_local;
          tc_fence_after();
          for (int j = 0; j < ntile && ok; ++j) {
            uint32_t g = it + j;
            int s3 = g % NKB, b = g & 1;
            if (!mbar_wait(&sm.k_full[s3], (g / NKB) & 1, kWait, abort_flag) ||
                (g >= 2 && !mbar_wait(&sm.s_empty[b], ((g >> 1) - 1) & 1, kWait, abort_flag))) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_qk(tm, sm.q, sm.k[s3], b);
            mma_commit(&sm.s_full[b]);
            mma_commit(&sm.k_empty[s3]);
            if (j + 1 == ntile) mma_commit(&sm.q_empty);  // every Q K^T of this item is issued
          }
          it += ntile;
        }
        if (*abort_flag) {
          mma_commit(&sm.drain2);  // every MMA issued by this thread has completed
          mbar_wait_drain(&sm.drain2, 0, kWait);
        }
      }
    }
  } else if (warp < 8) {
    // ------------------------------------------------------------ softmax (warps 4..7)
    regs_dec<112>();  // below the launch's 128: a decrease
    const int wq = warp & 3;
    const int row = wq * 32 + lane;
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    uint32_t it = 0;
    int po_seen = 0;
    float S_cur = 0.0f;
    int n_cur = 0;
    bool ok = true;
    for (int item = cta; item < n_items && ok; item += ncta) {
      ItemB bi = decode_b(L, item);
      if (bi.nslot == 0) continue;
      const TcTraj &tr = L.t[bi.t];
      int rows = L.g * tr.W;
      int grow = bi.rt * BM + row;
      bool valid_row = grow < rows;
      int qp = -0x7fffffff;
      // the row stats of this slice are complete once every share is merged
      if (FUSED && !warp_poll_geq(&L.merged[slice_of(L, bi)], 4u * items_per_slice(L, bi.t), abort_flag, hdr)) {
        ok = false;
        break;
      }
      // rows outside the slice, or rows that see nothing, get e = 0 everywhere
      float neg_m2 = -INFINITY;
      if (valid_row) {
        int h = bi.kvh * L.g + grow / tr.W, w = grow % tr.W;
        qp = tr.qpos[w];
        float mn = tr.stats[(((int64_t)bi.l * L.Hq + h) * tr.W + w) * (D + 4)];
        if (mn != -INFINITY) neg_m2 = -mn * 1.4426950408889634f;
      }
      int ntile = (bi.nslot + SLOTS - 1) / SLOTS;
      for (int j = 0; j < ntile && ok; ++j) {
        uint32_t g = it + j;
        int s = g % NKB, b = g & 1;
        // the slot table of this stage is published with its K copies (warp-
        // uniform results keep the lanes together for the collective ops)
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.k_full[s], (g / NKB) & 1, kWait, abort_flag))) {
          ok = false;
          break;
        }
        // slots inside the prefix every probe row sees need no position test
        const bool full = sm.tile_full[s] != 0;
        if (!full) {  // each warp keeps its own copy: no cross-warp barrier
          __syncwarp();
#pragma unroll 1
          for (int c = lane; c < BT; c += 32) {
            const SlotMeta mt = sm.meta[s][c / SLOT];
            int i = c % SLOT;
            sm.pos[wq][c] = i < mt.nv ? tr.pos[mt.tok0 + i] : 0x7fffffff;
          }
          __syncwarp();
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[b], (g >> 1) & 1, kWait, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        // Per 32-column chunk (two slots): e = exp(s - m) on the visible page
        // tokens (a visibility bit mask turns the others into -inf, so e = 0);
        // P as the (hi, lo) bf16 pair written over the S columns just read;
        // slot sums accumulate into page sums S_E, which go to the page FIFO
        // when the page's last slot is done.  The chunk loop is not unrolled:
        // a small loop body keeps the instruction cache warm.
        const int po_first = po_seen;
#pragma unroll 1
        for (int ch = 0; ch < BT / 32 && ok; ++ch) {
          float x[32];
          // tensor-memory loads and stores are warp-collective: the lanes
          // may have left the bounded waits above on different iterations
          __syncwarp();
          tmem_ld32f(tm + lane_base + b * BT + 32 * ch, x);
          const SlotMeta m0 = sm.meta[s][2 * ch], m1 = sm.meta[s][2 * ch + 1];
          uint32_t vm = (m0.nv >= SLOT ? 0xffffu : (1u << max(m0.nv, 0)) - 1u) |
                        ((m1.nv >= SLOT ? 0xffffu : (1u << max(m1.nv, 0)) - 1u) << 16);
          if (!full) {
#pragma unroll 1
            for (int i = 0; i < 32; ++i)
              if (sm.pos[wq][32 * ch + i] > qp) vm &= ~(1u << i);
          }
          if (!valid_row) vm = 0;
          tmem_wait_ld();
          float a0 = 0.f, a1 = 0.f, c0 = 0.f, c1 = 0.f;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            float xi = (vm >> i) & 1u ? x[i] : -INFINITY;
            x[i] = fast_exp2(fmaf(xi, L.scale_log2, neg_m2));
          }
#pragma unroll
          for (int i = 0; i < 16; i += 2) {
            a0 += x[i];
            a1 += x[i + 1];
            c0 += x[16 + i];
            c1 += x[17 + i];
          }
          uint32_t pk[32];
          split_pack32(x, pk);
          tmem_st32(tm + lane_base + b * BT + 32 * ch, pk);
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2) {
            const SlotMeta mt = h2 ? m1 : m0;
            if (mt.po < 0) continue;
            if (mt.flags & 1) {
              S_cur = 0.0f;
              n_cur = 0;
            }
            S_cur += h2 ? c0 + c1 : a0 + a1;
            n_cur += __popc(h2 ? vm >> 16 : vm & 0xffffu);
            if (mt.flags & 2) {
              int f = po_seen % NFIFO;
              if (!__all_sync(0xffffffffu, po_seen < NFIFO || mbar_wait(&sm.fifo_empty[f], ((po_seen / NFIFO) - 1) & 1,
                                                                           kWait, abort_flag))) {
                ok = false;
                break;
              }
              sm.fifo_s[f][row] = S_cur;
              sm.fifo_n[f][row] = n_cur;
              if (row == 0) sm.fifo_page[f] = sm.page_of[s][2 * ch + h2];
              ++po_seen;
            }
          }
        }
        __syncwarp();
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&sm.p_full[b]);
          // publish the pages this tile finished to the epilogue
          for (int k = po_first; k < po_seen; ++k) mbar_arrive(&sm.fifo_full[k % NFIFO]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.meta_empty[s]);  // done with the slot table
      }
      it += ntile;
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 8..15)
    // The two warpgroups take alternate pages: warpgroup 2 the even page
    // ordinals (accumulator U[0]), warpgroup 3 the odd ones (U[1]).  Each
    // thread owns one row and all 128 channels of that row's output o.
    regs_inc<168>();
    const int wq = warp & 3;
    const int par = (warp - 8) >> 2;
    const int row = wq * 32 + lane;
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    const uint32_t u_col = 2 * BT + par * D;
    int po = 0;
    bool ok = true;
    for (int item = cta; item < n_items && ok; item += ncta) {
      ItemB bi = decode_b(L, item);
      if (bi.nslot == 0) continue;
      const TcTraj &tr = L.t[bi.t];
      int rows = L.g * tr.W;
      int grow = bi.rt * BM + row;
      bool valid_row = grow < rows;
      int h = bi.kvh * L.g + (valid_row ? grow / tr.W : 0), w = valid_row ? grow % tr.W : 0;
      if (FUSED && !warp_poll_geq(&L.merged[slice_of(L, bi)], 4u * items_per_slice(L, bi.t), abort_flag, hdr)) {
        ok = false;
        break;
      }
      float2 o2[D / 2];
      float lsum = 0.0f, onorm = 0.0f;
      int nvis = 0;
      {
        const float *st = tr.stats + (((int64_t)bi.l * L.Hq + h) * tr.W + w) * (D + 4);
        float4 hd = valid_row ? *reinterpret_cast<const float4 *>(st) : make_float4(0.f, 0.f, 0.f, 0.f);
        lsum = hd.y;
        nvis = valid_row ? tr.nvis_w[w] : 0;
        float ss = 0.0f;
#pragma unroll
        for (int c = 0; c < D; c += 4) {
          float4 v = valid_row ? *reinterpret_cast<const float4 *>(st + 4 + c) : make_float4(0.f, 0.f, 0.f, 0.f);
          // explicit FMAs: the same rounding in every kernel this body is compiled into
          ss = fmaf(v.x, v.x, ss);
          ss = fmaf(v.y, v.y, ss);
          ss = fmaf(v.z, v.z, ss);
          ss = fmaf(v.w, v.w, ss);
          o2[c / 2] = make_float2(v.x, v.y);
          o2[c / 2 + 1] = make_float2(v.z, v.w);
        }
        onorm = sqrtf(ss);
      }
      int npages = tr.items[2 * bi.k + 1].x;
      for (int k = 0; k < npages && ok; ++k, ++po) {
        if ((po & 1) != par) continue;
        int f = po % NFIFO;
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.fifo_full[f], (po / NFIFO) & 1, kWait, abort_flag) &&
                                         mbar_wait(&sm.acc_full[par], (po >> 1) & 1, kWait, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        float S_E = sm.fifo_s[f][row];
        int n_E = sm.fifo_n[f][row];
        int E = sm.fifo_page[f];
        const float2 nS = make_float2(-S_E, -S_E);
        // ||U_E - S_E o||^2 over 16-column pieces of U_E
        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 16) {
          uint32_t r[16];
          tmem_ld16(tm + lane_base + u_col + c0, r);
          tmem_wait_ld();
          if (c0 + 16 == D) {  // U_E is in registers: hand the accumulator back
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
              mbar_arrive(&sm.acc_empty[par]);
              mbar_arrive(&sm.fifo_empty[f]);
            }
          }
#pragma unroll
          for (int i = 0; i < 16; i += 4) {
            float2 d0 = ffma2(nS, o2[(c0 + i) / 2], make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])));
            float2 d1 = ffma2(nS, o2[(c0 + i) / 2 + 1], make_float2(__uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])));
            acc0 = ffma2(d0, d0, acc0);
            acc1 = ffma2(d1, d1, acc1);
          }
        }
        float num2 = (acc0.x + acc0.y) + (acc1.x + acc1.y);
        float r = valid_row ? effect_value(n_E, nvis, S_E, lsum, num2, onorm) : 0.0f;
        if (valid_row && tr.headR) atomic_max_nonneg(tr.headR + ((int64_t)bi.l * L.Hq + h) * tr.P + E, r);
        float rm = r;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) rm = fmaxf(rm, __shfl_xor_sync(0xffffffffu, rm, off));
        if (lane == 0) atomic_max_nonneg(tr.R + E, rm);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tm, 512);
  if (threadIdx.x == 0 && sm.abort_flag) {
    if (FUSED) atomicExch(&hdr->abort, 1);
    record_error(hdr, COMMITKV_ERR_TIMEOUT, 11);
  }
}

__global__ void __launch_bounds__(512, 1) pass_b_tc(const __grid_constant__ TcLaunch L, WsHeader *hdr) {
  extern __shared__ uint8_t smem_raw[];
  page_body<false>(L, hdr, smem_raw, blockIdx.x, gridDim.x);
}

// ============================================================== fused
// One cooperative launch over all SMs: CTAs [0, n_a) run the flash pass
// (and merge the row stats slice by slice), CTAs [n_a, grid) run the page
// pass, each page-pass item waiting until its slice's stats are merged.
// Items of both passes are taken in slice order, so the page pass re-reads
// a slice's keys and values shortly after the flash pass read them, while
// they are still in L2.  Every cross-CTA wait is bounded.
__global__ void __launch_bounds__(512, 1) score_fused_tc(const __grid_constant__ TcLaunch L, WsHeader *hdr) {
  extern __shared__ uint8_t smem_raw[];
  if ((int)blockIdx.x < L.n_a) flash_body<true>(L, hdr, smem_raw, blockIdx.x, L.n_a);
  else page_body<true>(L, hdr, smem_raw, blockIdx.x - L.n_a, gridDim.x - L.n_a);
}


// ============================================================== host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool map_q(CUtensorMap *m, const void *q, uint64_t rows) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)D, rows};
  cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  cuuint32_t box[2] = {64, BM};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(q), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool map_kv(CUtensorMap *m, const void *base, int S, int H, int M, int64_t st, int64_t sh, int64_t sl,
            int box_rows) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)(S > 0 ? S : 1), (cuuint64_t)H, (cuuint64_t)M};
  cuuint64_t strides[3] = {(cuuint64_t)st * 2, (cuuint64_t)sh * 2, (cuuint64_t)sl * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)box_rows, 1, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

size_t smem_a() { return sizeof(SmemA) + 1024; }
size_t smem_b() { return sizeof(SmemB) + 1024; }

bool build_maps(TcMaps &mp, const TrajDev &t, int M, int H, int Hq) {
  uint64_t qrows = (uint64_t)M * Hq * (uint64_t)(t.W > 0 ? t.W : 1);
  bool ok = map_q(&mp.q, t.q, qrows) && map_kv(&mp.k, t.k, t.S, H, M, t.st, t.sh, t.sl, BT) &&
            map_kv(&mp.v, t.v, t.S, H, M, t.st, t.sh, t.sl, BT);
  for (int i = 0; i < 3 && ok; ++i)
    ok = map_kv(&mp.kb[i], t.k, t.S, H, M, t.st, t.sh, t.sl, SLOT << i) &&
         map_kv(&mp.vb[i], t.v, t.S, H, M, t.st, t.sh, t.sl, SLOT << i);
  return ok;
}

int fused_chunk_len(int max_tokens, int max_row_tiles) {
  // about kFusedItemsPerSlice flash items per slice (row tiles included), at
  // least 512 tokens each, whole 128-token tiles
  const int64_t per = ((int64_t)max_tokens * max_row_tiles + kFusedItemsPerSlice - 1) / kFusedItemsPerSlice;
  const int64_t c = per < 512 ? 512 : per;
  return (int)((c + BT - 1) / BT * BT);
}

int fused_flash_ctas(const TcLaunch &L, int sm_count) {
  int na = (int)(sm_count * kFusedFlashShare + 0.5);
  if (const char *e = getenv("COMMITKV_FUSED_FLASH_CTAS")) na = atoi(e);  // tuning experiments
  const int items_a = L.item_off_a[L.n_traj], items_b = L.item_off_b[L.n_traj];
  if (items_b == 0) na = sm_count;
  na = na < 1 ? 1 : na > sm_count - 1 ? sm_count - 1 : na;
  // A partial slot is reused n_a * kRing items later, after the slice of its
  // earlier item is merged.  That slice's items must all come earlier than
  // the reusing item (else the wait could depend on itself): n_a * kRing
  // must cover the items of any slice.
  int nis_max = 1;
  for (int t = 0; t < L.n_traj; ++t) {
    const int nis = L.t[t].nchunk * L.t[t].nrt;
    nis_max = nis > nis_max ? nis : nis_max;
  }
  const int na_min = (nis_max + kRing - 1) / kRing;
  na = na < na_min ? na_min : na;
  return na < items_a ? na : items_a;
}

cudaError_t launch_score_tc(TcLaunch &L, WsHeader *hdr, cudaStream_t s, int sm_count) {
  cudaError_t e;
  for (int t = 0; t < L.n_traj; ++t)
    if (L.t[t].nchunk > 32) return cudaErrorInvalidValue;  // the row merge takes at most 64 partials
  const int na_items = L.from_stats ? 0 : L.item_off_a[L.n_traj];
  const int nb_items = L.item_off_b[L.n_traj];
  if (L.fused && na_items > 0) {
    // fused: prep, then one cooperative launch of both passes
    const size_t smem = smem_a() > smem_b() ? smem_a() : smem_b();
    e = cudaFuncSetAttribute(score_fused_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_fused_tc, 512, smem);
    if (e != cudaSuccess) return e;
    if (per_sm != 1) return cudaErrorInvalidConfiguration;  // one CTA per SM: all 512 TMEM columns each
    L.n_a = fused_flash_ctas(L, sm_count);
    int nb = sm_count - L.n_a;
    nb = nb < nb_items ? nb : nb_items;
    if (nb < 1 && nb_items > 0) return cudaErrorInvalidConfiguration;
    prep_kernel<<<L.n_traj, 1024, 0, s>>>(L, hdr);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaMemsetAsync(L.a_done, 0, (size_t)L.slice_off[L.n_traj] * kCounterStride * 4, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(L.merged, 0, (size_t)L.slice_off[L.n_traj] * kCounterStride * 4, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(&hdr->abort, 0, sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    void *args[] = {(void *)&L, (void *)&hdr};
    return cudaLaunchCooperativeKernel((const void *)score_fused_tc, dim3(L.n_a + nb), dim3(512), args, smem, s);
  }
  e = cudaFuncSetAttribute(pass_a_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_a());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(pass_b_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_b());
  if (e != cudaSuccess) return e;
  prep_kernel<<<L.n_traj, 1024, 0, s>>>(L, hdr);
  if (na_items > 0) pass_a_tc<<<na_items < sm_count ? na_items : sm_count, 384, smem_a(), s>>>(L, hdr);
  const int rows = L.from_stats ? 0 : L.row_off[L.n_traj];
  if (rows > 0) combine_tc<<<(rows * 32 + 255) / 256, 256, 0, s>>>(L);
  if (nb_items > 0) pass_b_tc<<<nb_items < sm_count ? nb_items : sm_count, 512, smem_b(), s>>>(L, hdr);
  return cudaGetLastError();
}

}  // namespace tc
}  // namespace ckv
