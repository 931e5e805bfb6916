// Greedy joint test (Section 3.3, Eq. 11) on the 5th-generation tensor
// cores: bf16 K/V/Q, head_dim 128, fp32 accumulation in tensor memory.
//
// One cooperative persistent kernel, one CTA of 256 threads per SM.  A
// group is 128 probe rows of one (trajectory, selected layer, KV head), TMEM
// lane i holding row i; the CTA's threads form two teams of four warps, and
// thread i of each team works on row i: the teams split the pages in the
// softmax and the channels in the epilogue.  In every round (joint_common.cuh) a
// group makes up to two passes of the same machinery over a list of at
// most four pages:
//   fold  the pages of the previous round that were accepted: their D_E are
//         computed again (bit-identical to the values that round used) and
//         added, in candidate order, into the row's D_A, S_A, n_A in the
//         workspace;
//   scan  the round's candidates: Eq. 6 on A u T for every non-empty subset
//         T of them, max over the rows (Eq. 7) into the round's table.
// A pass stages Q (once per group and round) and the pages' K and V rows in
// shared memory (cp.async into the 128-byte-swizzled layout) and issues
//   S = Q K^T       one MMA chain with N = 32 x pages, TMEM columns 256..383
//   e = exp(s - m)  per row on the page's visible tokens (m = the row's
//                   final max); S_E = sum e, n_E = count; P = e written
//                   over S as a bf16 (hi, lo) pair
//   U_E = P V_E     per page and 64-channel half, TMEM columns 64 c, TS form
//                   (P from tensor memory, V from shared memory)
// and the epilogue reads U_E 8 columns at a time (o and D_A of the channel
// half staged in shared memory while the MMAs run): D_E = U_E - S_E o.  In
// the scan the sums of the subsets are built as a tree in which every
// subset adds its largest page last, so each is the sum that the
// one-page-at-a-time scan forms, ((D_A + D_b1) + D_b2) + ... + D_c, and its
// squared norm accumulates over the channels in order.
// Pages longer than 32 tokens are taken in 32-token chunks: U accumulates
// over the chunks, and the chunks' QK and softmax are redone for the second
// channel half.  Every mbarrier wait is bounded (1 s); on expiry the kernel
// records COMMITKV_ERR_TIMEOUT, raises the abort flag that the grid barrier
// watches, waits (bounded) for its MMAs in flight, frees its tensor memory
// and returns.
#include "joint_common.cuh"
#include "sm103.cuh"

namespace ckv {
namespace {

using namespace ckv::sm103;
using joint::kCombos;
using joint::kRound;

constexpr int D = 128;
constexpr int kRows = 128;   // probe rows per group (MMA M, TMEM lanes)
constexpr int kCT = 32;      // page tokens per chunk (the QK N of one page)
constexpr int kTeam = 128;                 // threads per team (one per row)
constexpr int kThreads = 2 * kTeam;
constexpr uint64_t kWait = 1000000000ull;
constexpr uint32_t kQHalf = kRows * 128;         // one 64-channel half of the Q tile: 16 KB
constexpr uint32_t kKHalf = kRound * kCT * 128;  // K rows of all pages, one half: 16 KB
constexpr uint32_t kVHalf = kCT * 128;           // V rows of one page, one half: 4 KB
constexpr uint32_t kColS = 256;                  // TMEM column of page 0's S/P (kCT per page)
constexpr int kHalfPad = 68;                     // floats per row of the o / D_A half buffers
constexpr int kCached = 2;                       // groups per block whose row data stays in shared memory

struct SmemJ {
  alignas(1024) uint8_t q[2 * kQHalf];
  alignas(1024) uint8_t k[2 * kKHalf];
  alignas(1024) uint8_t v[kRound][2 * kVHalf];
  // o and D_A of one 64-channel half of every row (each thread its own
  // row; the padding keeps the rows' 16-byte words in distinct banks)
  alignas(16) float oh[kRows][kHalfPad];
  alignas(16) float dah[kRows][kHalfPad];
  float Sc[kRound][kRows];     // S_E of every page and row (written by the page's team)
  int nc[kRound][kRows];       // n_E
  float part[kCombos + 1][kRows];  // team 1's sums of squares (and ||o||^2) for team 0
  float part2[kCombos / 2 + 1][kRows];  // team 0's, for the subsets that team 1 evaluates
  // the row data of the block's first kCached groups, kept from round to
  // round: final max (base 2), exp-sum, visible count, position, S_A, n_A
  float rc_m2[kCached][kRows], rc_l[kCached][kRows], rc_SA[kCached][kRows];
  int rc_nvis[kCached][kRows], rc_qp[kCached][kRows], rc_nA[kCached][kRows];
  int pos[kRound][kCT];
  unsigned rmax[16];
  uint64_t bar;       // Q K^T done (one issuing thread)
  uint64_t bar_pv;    // P V done (two issuing threads)
  uint64_t drain[2];  // an issuing thread's MMAs done (after an abort)
  uint32_t tmem;
  int abort_flag;
};

struct Group {
  int t, l, li, kvh, rows, row0;
};

// What a thread keeps of its probe row.
struct Row {
  bool ok;          // inside the group
  int64_t grow;     // index into D_A, S_A
  const float *st;  // stats row: m, l, n, pad, o[D]
  float m2, l;      // final max in base-2 units, exp-sum
  int nvis, qp;
  float SA;
  int nA;
};

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// K-major tile of 128-byte rows in two 64-channel halves half_bytes apart:
// the descriptor of k-step ks (16 channels).
__device__ __forceinline__ uint64_t desc_kmajor(const uint8_t *tile, uint32_t half_bytes, int ks) {
  return smem_desc(smem_addr(tile) + (ks >> 2) * half_bytes + (ks & 3) * 32, 16, 1024, kSwizzle128B);
}
// V rows of one page as the MN-major B operand (k = tokens, n = the 64
// channels of half h): k-step ks (16 tokens).
__device__ __forceinline__ uint64_t desc_v(const uint8_t *tile, int h, int ks) {
  return smem_desc(smem_addr(tile) + h * kVHalf + ks * 2048, kVHalf, 1024, kSwizzle128B);
}
// TMEM column of the 8 packed P columns (hi or lo) of page c, k-step ks.
__device__ __forceinline__ uint32_t p_col(int c, int ks, int lo) {
  return kColS + kCT * c + 32 * (ks >> 1) + 8 * (ks & 1) + 16 * lo;
}
static_assert(kCT == 32, "one 32-column TMEM load covers a page chunk's scores");

__device__ __forceinline__ Group decode_group(const JointLaunch &L, int grp) {
  const Batch &b = L.batch;
  Group G;
  G.t = joint::find_group_traj(L.group_off, b.n_traj, grp);
  int local = grp - L.group_off[G.t], nrb = L.nrb[G.t];
  const int rb = local % nrb;
  local /= nrb;
  G.kvh = local % b.H;
  G.li = local / b.H;
  G.l = b.layer_ids[G.li];
  G.rows = b.g * b.t[G.t].W;
  G.row0 = rb * kRows;
  return G;
}

// Waits for the MMAs committed to a pass barrier; uniform over the block.
__device__ __forceinline__ bool wait_mma(SmemJ &s, uint64_t *bar, uint32_t &phase) {
  bool ok = mbar_wait(bar, phase, kWait, &s.abort_flag);
  phase ^= 1u;
  ok = __syncthreads_and(ok) != 0;
  if (ok) tc_fence_after();
  return ok;
}

constexpr int kSub = 8;  // channels per epilogue step

// Starts the copies of o and D_A of the team's 32 channels of half h of the
// thread's row into that row of the half buffers.
__device__ __forceinline__ void stage_half(SmemJ &s, const Row &rw, const float *DA, int h) {
  if (!rw.ok) return;
  const int i = threadIdx.x % kTeam, c0 = 32 * (threadIdx.x / kTeam);
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    cp_async16(&s.oh[i][c0 + 4 * u], rw.st + 4 + 64 * h + c0 + 4 * u);
    cp_async16(&s.dah[i][c0 + 4 * u], DA + rw.grow * D + 64 * h + c0 + 4 * u);
  }
}

// 32 lanes x 8 consecutive 32-bit columns.
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[kSub]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
}

// Largest member of the non-empty set T (a constant after unrolling).
__host__ __device__ constexpr int top_bit(int T) { return T >= 8 ? 3 : T >= 4 ? 2 : T >= 2 ? 1 : 0; }

// One pass over the pages list[0..n) (n <= kRound).  kScan: accumulates the
// squared norms of the subset sums over the team's channels into ss, and
// o's into on2 (even and odd channels apart); otherwise adds the pages' D_E into D_A in the workspace.
// S_E and n_E of every page are left in Sc and nc.  Returns false on a
// timeout.
template <bool kScan>
__device__ __forceinline__ bool run_pass(SmemJ &s, const JointLaunch &L, WsHeader *hdr, const Group &G,
                                         const Row &rw, const int *list, int n, bool stage_q, uint32_t tm,
                                         uint32_t lane_base, uint32_t &phase, uint32_t &phase_pv,
                                         float2 (&ss)[kCombos], float2 &on2,
                                         float (&Sc)[kRound], int (&nc)[kRound]) {
  const Batch &b = L.batch;
  const TrajDev &tr = b.t[G.t];
  const int tid = threadIdx.x, team = tid / kTeam, r = tid % kTeam;
  int ps[kRound], pl[kRound];
  int nch = 1;
#pragma unroll
  for (int c = 0; c < kRound; ++c) {
    ps[c] = pl[c] = 0;
    Sc[c] = 0.0f;
    nc[c] = 0;
    if (c < n) {
      const int E = list[c];
      if (E < 0 || E >= tr.P) {
        if (tid == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -4);
      } else {
        ps[c] = tr.ps[E];
        pl[c] = tr.pl[E];
        if (pl[c] < 0 || ps[c] < 0 || ps[c] > tr.S - pl[c]) {
          if (tid == 0) record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, E);
          ps[c] = pl[c] = 0;
        }
      }
      nch = max(nch, (pl[c] + kCT - 1) / kCT);
    }
  }
  const __nv_bfloat16 *kp =
      static_cast<const __nv_bfloat16 *>(tr.k) + (int64_t)G.l * tr.sl + (int64_t)G.kvh * tr.sh;
  const __nv_bfloat16 *vp =
      static_cast<const __nv_bfloat16 *>(tr.v) + (int64_t)G.l * tr.sl + (int64_t)G.kvh * tr.sh;

  for (int h = 0; h < 2; ++h) {
    for (int j = 0; j < nch; ++j) {
      int nt[kRound];
#pragma unroll
      for (int c = 0; c < kRound; ++c) nt[c] = c < n ? min(kCT, max(0, pl[c] - j * kCT)) : 0;
      if (h == 0 || nch > 1) {
        // ---- stage (the MMAs that read the buffers have completed)
        __syncthreads();
        if (stage_q && h == 0 && j == 0) {
          for (int e = tid; e < kRows * 16; e += kThreads) {
            const int r = e >> 4, k16 = e & 15, row = G.row0 + r;
            if (row < G.rows) {
              const int hq = G.kvh * b.g + row / tr.W, w = row % tr.W;
              const __nv_bfloat16 *src =
                  static_cast<const __nv_bfloat16 *>(tr.q) + (((int64_t)G.l * b.Hq + hq) * tr.W + w) * D + 8 * k16;
              cp_async16(s.q + (k16 >> 3) * kQHalf + sw128_offset(r, k16 & 7), src);
            }
          }
        }
        for (int e = tid; e < n * kCT * 16; e += kThreads) {
          const int c = e / (kCT * 16), rem = e % (kCT * 16), i = rem >> 4, k16 = rem & 15;
          if (i < nt[c]) {
            const int64_t off = (int64_t)(ps[c] + j * kCT + i) * tr.st + 8 * k16;
            cp_async16(s.k + (k16 >> 3) * kKHalf + sw128_offset(kCT * c + i, k16 & 7), kp + off);
            cp_async16(s.v[c] + (k16 >> 3) * kVHalf + sw128_offset(i, k16 & 7), vp + off);
          }
        }
        for (int e = tid; e < n * kCT; e += kThreads) {
          const int c = e / kCT, i = e % kCT;
          s.pos[c][i] = i < nt[c] ? tr.pos[ps[c] + j * kCT + i] : 0;
        }
        cp_async_wait_all();
        fence_proxy_async();
        __syncthreads();
        // ---- S = Q K^T for all pages of the pass
        if (tid == 0) {
          tc_fence_after();
          const uint32_t idesc = idesc_bf16_f32(kRows, kCT * n, 0, 0);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks)
            mma_bf16(tm + kColS, desc_kmajor(s.q, kQHalf, ks), desc_kmajor(s.k, kKHalf, ks), idesc, ks > 0);
          mma_commit(&s.bar);
        }
        if (!wait_mma(s, &s.bar, phase)) return false;
        // ---- e = exp(s - m) on the visible tokens; P over S (team t takes
        // the pages c = t mod 2)
#pragma unroll 1
        for (int c = team; c < n; c += 2) {
          float x[32];
          uint32_t pk[32];
          const uint32_t addr = tm + lane_base + kColS + kCT * c;
          tmem_ld32f(addr, x);
          tmem_wait_ld();
          // the chunk's visible tokens: positions increase along the page,
          // so they are a prefix, whole unless the row's position cuts it
          int ne = 0;
          if (rw.ok && nt[c] > 0) {
            if (s.pos[c][nt[c] - 1] <= rw.qp) {
              ne = nt[c];
            } else {
#pragma unroll 1
              for (int i = 0; i < nt[c]; ++i) ne += s.pos[c][i] <= rw.qp ? 1 : 0;
            }
          }
          float se = 0.0f;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float e = i < ne ? fast_exp2(fmaf(x[i], b.scale_log2, -rw.m2)) : 0.0f;
            se += e;
            x[i] = e;
          }
          if (h == 0) {
            Sc[c] += se;
            nc[c] += ne;
            s.Sc[c][r] = Sc[c];
            s.nc[c][r] = nc[c];
          }
          split_pack32(x, pk);
          tmem_st32(addr, pk);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncthreads();
      }
      // ---- U_E (+)= P V_E for channel half h; two threads issue, the even
      // and the odd pages (accumulators of their own), and both commit
      if (tid == 0 || tid == 32) {
        tc_fence_after();
        const uint32_t idesc = idesc_bf16_f32(kRows, 64, 0, 1);
#pragma unroll 1
        for (int c = tid / 32; c < n; c += 2) {
          const int nks = max(1, (nt[c] + 15) / 16);
#pragma unroll 1
          for (int ks = 0; ks < nks; ++ks) {
            const uint64_t bd = desc_v(s.v[c], h, ks);
            mma_bf16_ts(tm + 64 * c, tm + p_col(c, ks, 0), bd, idesc, (j > 0 || ks > 0) ? 1u : 0u);
            mma_bf16_ts(tm + 64 * c, tm + p_col(c, ks, 1), bd, idesc, 1u);
          }
        }
        mma_commit(&s.bar_pv);
      }
      const bool last = j == nch - 1;
      if (last) stage_half(s, rw, L.DA, h);  // in flight while the MMAs run
      if (!wait_mma(s, &s.bar_pv, phase_pv)) return false;
      if (last) {
        cp_async_wait_all();  // the thread's own parts of the half buffers
        if (h == 0) {
#pragma unroll
          for (int c = 0; c < kRound; ++c)
            if (c < n) {
              Sc[c] = s.Sc[c][r];
              nc[c] = s.nc[c][r];
            }
        }
        // ---- epilogue over the team's 32 channels of half h, kSub at a time
#pragma unroll 1
        for (int q = 4 * team; q < 4 * team + 4; ++q) {
          const int ch0 = 64 * h + kSub * q;
          float o[kSub], da[kSub];
#pragma unroll
          for (int u4 = 0; u4 < kSub / 4; ++u4) {
            const float4 x = *reinterpret_cast<const float4 *>(&s.oh[r][kSub * q + 4 * u4]);
            const float4 y = *reinterpret_cast<const float4 *>(&s.dah[r][kSub * q + 4 * u4]);
            o[4 * u4] = x.x, o[4 * u4 + 1] = x.y, o[4 * u4 + 2] = x.z, o[4 * u4 + 3] = x.w;
            da[4 * u4] = y.x, da[4 * u4 + 1] = y.y, da[4 * u4 + 2] = y.z, da[4 * u4 + 3] = y.w;
          }
          uint32_t u[kRound][kSub];
#pragma unroll
          for (int c = 0; c < kRound; ++c)
            if (c < n) tmem_ld8(tm + lane_base + 64 * c + kSub * q, u[c]);
          tmem_wait_ld();
          // two channels per packed instruction (an addition as a product
          // with 1: the same rounding)
          const float2 one2 = make_float2(1.0f, 1.0f);
#pragma unroll
          for (int i = 0; i < kSub; i += 2) {
            const float2 o2 = make_float2(o[i], o[i + 1]);
            float2 de[kRound];
#pragma unroll
            for (int c = 0; c < kRound; ++c)
              de[c] = c < n ? ffma2(make_float2(-Sc[c], -Sc[c]), o2,
                                    make_float2(__uint_as_float(u[c][i]), __uint_as_float(u[c][i + 1])))
                            : make_float2(0.0f, 0.0f);
            if constexpr (kScan) {
              on2 = ffma2(o2, o2, on2);
              float2 p[1 << kRound];
              p[0] = make_float2(da[i], da[i + 1]);
#pragma unroll
              for (int T = 1; T < (1 << kRound); ++T) {
                if (T >= (1 << n)) break;  // subsets of the pass's pages only
                p[T] = ffma2(de[top_bit(T)], one2, p[T & ~(1 << top_bit(T))]);
                ss[T - 1] = ffma2(p[T], p[T], ss[T - 1]);
              }
            } else {
              float2 x = make_float2(da[i], da[i + 1]);
#pragma unroll
              for (int c = 0; c < kRound; ++c)
                if (c < n) x = ffma2(de[c], one2, x);
              da[i] = x.x;
              da[i + 1] = x.y;
            }
          }
          if constexpr (!kScan) {
            if (rw.ok) {
              float4 *pa = reinterpret_cast<float4 *>(L.DA + rw.grow * D + ch0);
#pragma unroll
              for (int u4 = 0; u4 < kSub / 4; ++u4)
                pa[u4] = make_float4(da[4 * u4], da[4 * u4 + 1], da[4 * u4 + 2], da[4 * u4 + 3]);
            }
          }
        }
        if constexpr (!kScan) __threadfence();  // D_A is read again through L2 by the scan
      }
      // the epilogue's TMEM reads are done before the next MMAs write
      tc_fence_before();
      __syncthreads();
    }
  }
  return true;
}

__global__ void __launch_bounds__(kThreads, 1) joint_tc_kernel(const __grid_constant__ JointLaunch L,
                                                             WsHeader *hdr) {
  extern __shared__ uint8_t smem_raw[];
  SmemJ &s = *reinterpret_cast<SmemJ *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Batch &b = L.batch;
  const int tid = threadIdx.x, warp = tid / 32, lane = tid % 32;

  // Rows past a page's end are never written: they keep finite values (zero
  // or an earlier page's), whose scores are masked and whose V rows meet
  // P = 0.
  for (int i = tid; i < (int)(sizeof(s.q) / 16); i += kThreads) reinterpret_cast<uint4 *>(s.q)[i] = uint4{};
  for (int i = tid; i < (int)(sizeof(s.k) / 16); i += kThreads) reinterpret_cast<uint4 *>(s.k)[i] = uint4{};
  for (int i = tid; i < (int)(sizeof(s.v) / 16); i += kThreads) reinterpret_cast<uint4 *>(&s.v[0][0])[i] = uint4{};
  for (int i = tid; i < kRows * kHalfPad; i += kThreads) (&s.oh[0][0])[i] = (&s.dah[0][0])[i] = 0.0f;
  if (tid == 0) {
    s.abort_flag = 0;
    mbar_init(&s.bar, 1);
    mbar_init(&s.bar_pv, 2);
    mbar_init(&s.drain[0], 1);
    mbar_init(&s.drain[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&s.tmem, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = s.tmem;
  // warps w and w + 4 (the two teams) reach TMEM lanes 32 (w mod 4) ..
  const uint32_t lane_base = (uint32_t)((warp % 4) * 32) << 16;
  uint32_t phase = 0, phase_pv = 0;
  bool ok = true;

  const int rounds = joint::round_total(L);
  const int ngroups = L.group_off[b.n_traj];
  for (int r = 0; r < rounds && ok; ++r) {
    float *tab_r = joint::round_table(L, r);
    for (int grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
      const Group G = decode_group(L, grp);
      const TrajDev &tr = b.t[G.t];
      const int kc = joint::round_count(L, G.t, r);
      if (kc == 0) continue;
      // the previous round's accepted pages, in candidate order
      int fold[kRound], nf = 0;
      if (r > 0) {
        const int kp = joint::round_count(L, G.t, r - 1);
        const unsigned acc =
            joint::resolve_round(joint::round_table(L, r - 1) + G.t * kCombos, kp, L.tau);
        for (int c = 0; c < kp; ++c)
          if ((acc >> c) & 1u) fold[nf++] = L.cand[G.t][(r - 1) * kRound + c];
      }
      int cand[kRound];
      for (int c = 0; c < kc; ++c) cand[c] = L.cand[G.t][r * kRound + c];

      Row rw;
      const int row = G.row0 + tid % kTeam;
      rw.ok = row < G.rows;
      const int hq = G.kvh * b.g + (rw.ok ? row / tr.W : 0), w = rw.ok ? row % tr.W : 0;
      rw.grow = L.row_off[G.t] + (int64_t)(G.li * b.H + G.kvh) * G.rows + (rw.ok ? row : 0);
      rw.st = L.stats[G.t] + (((int64_t)G.l * b.Hq + hq) * tr.W + w) * (D + 4);
      // the block's k-th group; its row data is read from global memory in
      // the first round and from the shared copy after that
      const int kslot = (grp - (int)blockIdx.x) / (int)gridDim.x, rr = tid % kTeam;
      if (kslot < kCached && r > 0) {
        rw.m2 = s.rc_m2[kslot][rr];
        rw.l = s.rc_l[kslot][rr];
        rw.nvis = s.rc_nvis[kslot][rr];
        rw.qp = s.rc_qp[kslot][rr];
        rw.SA = s.rc_SA[kslot][rr];
        rw.nA = s.rc_nA[kslot][rr];
      } else {
        const float mn = rw.ok ? rw.st[0] : -__builtin_huge_valf();
        rw.m2 = mn == -__builtin_huge_valf() ? mn : mn * 1.4426950408889634f;
        rw.l = rw.ok ? rw.st[1] : 0.0f;
        rw.nvis = rw.ok ? (int)rw.st[2] : 0;
        rw.qp = rw.ok ? tr.qpos[w] : -0x7fffffff;
        rw.SA = rw.ok ? L.SA[rw.grow * 2] : 0.0f;
        rw.nA = rw.ok ? (int)L.SA[rw.grow * 2 + 1] : 0;
      }
      if (tid < 16) s.rmax[tid] = 0u;

      float2 ss2[kCombos], on2p = make_float2(0.0f, 0.0f);
      float Sc[kRound];
      int nc[kRound];
#pragma unroll
      for (int i = 0; i < kCombos; ++i) ss2[i] = make_float2(0.0f, 0.0f);
      if (nf > 0) {
        if (!run_pass<false>(s, L, hdr, G, rw, fold, nf, true, tm, lane_base, phase, phase_pv, ss2, on2p, Sc,
                             nc)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int c = 0; c < kRound; ++c)
          if (c < nf) {
            rw.SA += Sc[c];
            rw.nA += nc[c];
          }
        if (rw.ok && tid < kTeam) {
          L.SA[rw.grow * 2] = rw.SA;
          L.SA[rw.grow * 2 + 1] = (float)rw.nA;
        }
      }
      if (kslot < kCached && tid < kTeam) {  // read again by both teams in the next round
        s.rc_m2[kslot][rr] = rw.m2;
        s.rc_l[kslot][rr] = rw.l;
        s.rc_nvis[kslot][rr] = rw.nvis;
        s.rc_qp[kslot][rr] = rw.qp;
        s.rc_SA[kslot][rr] = rw.SA;
        s.rc_nA[kslot][rr] = rw.nA;
      }
      if (!run_pass<true>(s, L, hdr, G, rw, cand, kc, nf == 0, tm, lane_base, phase, phase_pv, ss2, on2p,
                          Sc, nc)) {
        ok = false;
        break;
      }
      // the channel sums of the thread; team 0 evaluates the subsets
      // T = 1..8 and team 1 the subsets T = 9..15, each with the other team's
      // sums of its channels added (one addition of two floats: the same
      // value in either order)
      constexpr int kSplit = kCombos / 2 + 1;  // subsets T <= kSplit go to team 0
      float ss[kCombos], on2 = on2p.x + on2p.y;
#pragma unroll
      for (int i = 0; i < kCombos; ++i) ss[i] = ss2[i].x + ss2[i].y;
      if (tid >= kTeam) {
#pragma unroll
        for (int i = 0; i < kSplit; ++i) s.part[i][rr] = ss[i];
        s.part[kCombos][rr] = on2;
      } else {
#pragma unroll
        for (int i = kSplit; i < kCombos; ++i) s.part2[i - kSplit][rr] = ss[i];
        s.part2[kCombos - kSplit][rr] = on2;
      }
      __syncthreads();
      {
        const int T0 = tid < kTeam ? 1 : kSplit + 1, T1 = tid < kTeam ? kSplit : kCombos;
        if (tid < kTeam) {
#pragma unroll
          for (int i = 0; i < kSplit; ++i) ss[i] += s.part[i][rr];
          on2 += s.part[kCombos][rr];
        } else {
#pragma unroll
          for (int i = kSplit; i < kCombos; ++i) ss[i] += s.part2[i - kSplit][rr];
          on2 += s.part2[kCombos - kSplit][rr];
        }
        // Eq. 6 on A u T for every non-empty subset T of the round's pages;
        // S and n added in candidate order
        const float onorm = sqrtf(on2);
#pragma unroll
        for (int T = 1; T < (1 << kRound); ++T) {
          if (T >= (1 << kc)) break;
          if (T < T0 || T > T1) continue;
          float S_tot = rw.SA;
          int n_tot = rw.nA;
#pragma unroll
          for (int c = 0; c < kRound; ++c)
            if ((T >> c) & 1) {
              S_tot += Sc[c];
              n_tot += nc[c];
            }
          const float rv = rw.ok ? effect_value(n_tot, rw.nvis, S_tot, rw.l, ss[T - 1], onorm) : 0.0f;
          const unsigned mx = __reduce_max_sync(0xffffffffu, __float_as_uint(rv));
          if (lane == 0) atomicMax(&s.rmax[T - 1], mx);
        }
      }
      __syncthreads();
      if (tid < (1 << kc) - 1) atomic_max_nonneg(tab_r + G.t * kCombos + tid, __uint_as_float(s.rmax[tid]));
    }
    if (!ok) break;
    if (!joint::grid_barrier(hdr, gridDim.x)) {
      ok = false;
      break;
    }
    if (blockIdx.x == 0) joint::publish_round(L, r);
  }

  if (!ok) {
    // a wait ran out (or another block gave up): leave the grid barrier to
    // the others and let the MMAs in flight finish before the memory goes
    if (tid == 0) {
      if (s.abort_flag) record_error(hdr, COMMITKV_ERR_TIMEOUT, -5);
      atomicExch(&hdr->abort, 1);
    }
    if (tid == 0 || tid == 32) {  // the issuing threads: every MMA of theirs has completed
      mma_commit(&s.drain[tid / 32]);
      mbar_wait_drain(&s.drain[tid / 32], 0, kWait);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
}

}  // namespace

// bf16, head_dim 128, and 16-byte aligned rows of K, V, Q and the stats.
bool joint_tc_eligible(const JointLaunch &L) {
  const Batch &b = L.batch;
  if (b.dtype != COMMITKV_BF16 || b.d != D) return false;
  for (int t = 0; t < b.n_traj; ++t) {
    const TrajDev &tr = b.t[t];
    if (tr.P == 0 || tr.W == 0) continue;
    if ((reinterpret_cast<uintptr_t>(tr.k) | reinterpret_cast<uintptr_t>(tr.v) |
         reinterpret_cast<uintptr_t>(tr.q) | reinterpret_cast<uintptr_t>(L.stats[t])) & 15)
      return false;
    if ((tr.sl | tr.sh | tr.st) & 7) return false;
  }
  return true;
}

int joint_tc_rows_per_group() { return kRows; }

cudaError_t launch_joint_tc(const JointLaunch &L, WsHeader *hdr, cudaStream_t stream, int sm_count) {
  const size_t smem = sizeof(SmemJ) + 1024;
  cudaError_t e = cudaFuncSetAttribute(joint_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, joint_tc_kernel, kThreads, smem);
  if (e != cudaSuccess) return e;
  // one CTA per SM: each takes all 512 TMEM columns
  if (per_sm != 1) return cudaErrorInvalidConfiguration;
  const int ngroups = L.group_off[L.batch.n_traj];
  const int grid = ngroups < sm_count ? ngroups : sm_count;
  if (grid < 1) return cudaSuccess;
  void *args[] = {(void *)&L, (void *)&hdr};
  return cudaLaunchCooperativeKernel((const void *)joint_tc_kernel, dim3(grid), dim3(kThreads), args, smem,
                                     stream);
}

}  // namespace ckv
