// Compression checkpoint (Section 3.3, Eq. 12-13) and the shared-index
// gather of keys, values and absolute positions (Eq. 4).
//
// select  one block per trajectory: mark retired tokens, protect the
//         pending prefix, pick the fill tokens by an exact radix select on
//         64-bit keys (fill score, token index), and write I_j ascending;
// gather  16-byte vector copies of the retained K and V rows of every
//         (layer, KV head), plus positions; into caller buffers, or in place
//         (the retained rows move to rows 0..|I|-1 of the cache itself).
#include <type_traits>

#include "ckv_internal.cuh"

namespace ckv {
namespace {

constexpr int kThreads = 1024;
constexpr int kMaxPending = 2048;

__device__ __forceinline__ uint64_t fill_key(float f, int i) {
  uint32_t u = __float_as_uint(f == 0.0f ? 0.0f : f);  // -0 and +0 tie
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);       // order-preserving
  return ((uint64_t)u << 32) | (uint32_t)i;              // ties: higher index first
}

// Block-wide exclusive scan of one int per thread; returns the total.
__device__ int block_scan(int v, int *excl, int *s_warp) {
  int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kThreads / 32 ? s_warp[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    s_warp[lane] = w;  // inclusive prefix of warp totals
  }
  __syncthreads();
  int before = warp ? s_warp[warp - 1] : 0;
  *excl = before + x - v;
  int total = s_warp[kThreads / 32 - 1];
  __syncthreads();
  return total;
}

__global__ void __launch_bounds__(kThreads, 1) select_kernel(const __grid_constant__ CompactLaunch L,
                                                          WsHeader *hdr) {
  int t = blockIdx.x;
  const TrajDev &tr = L.t[t];
  int S = tr.S, P = tr.P;
  uint8_t *cls = L.cls[t];  // 0 = fill candidate, 1 = retired, 2 = protected, 3 = kept
  __shared__ int s_warp[32];
  __shared__ int s_bad, s_prot_tokens, s_rem;
  __shared__ int s_pid[kMaxPending];
  __shared__ float s_pr[kMaxPending];
  __shared__ int s_order[kMaxPending];
  __shared__ uint8_t s_take[kMaxPending];
  __shared__ unsigned s_hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_krem, s_exact;

  if (threadIdx.x == 0) {
    s_bad = 0;
    s_prot_tokens = 0;
    s_rem = 0;
  }
  for (int i = threadIdx.x; i < S; i += kThreads) {
    cls[i] = 0;
    if (isnan(L.fill[t][i])) s_bad = 1;
  }
  __syncthreads();
  // retired pages (D_c) are excluded
  for (int E = threadIdx.x; E < P; E += kThreads) {
    int ps = tr.ps[E], pl = tr.pl[E];
    if (pl < 0 || ps < 0 || ps > S - pl) {
      s_bad = 1;
      continue;
    }
    if (L.retired[t][E])
      for (int i = ps; i < ps + pl; ++i) cls[i] = 1;
  }
  // pending pages: drop retired ones, order by (priority desc, page index asc)
  int np = L.n_pending[t];
  for (int k = threadIdx.x; k < np; k += kThreads) {
    int E = L.pending[t][k];
    float pr = (E >= 0 && E < P) ? L.prio[t][E] : 0.0f;
    if (E < 0 || E >= P || isnan(pr)) {
      s_bad = 1;
      E = -1;
    } else if (L.retired[t][E]) {
      E = -1;
    }
    s_pid[k] = E;
    s_pr[k] = pr;
  }
  __syncthreads();
  for (int k = threadIdx.x; k < np; k += kThreads) {
    int E = s_pid[k];
    if (E < 0) continue;
    float pr = s_pr[k];
    int rank = 0;
    for (int j = 0; j < np; ++j) {
      int F = s_pid[j];
      if (F < 0) continue;
      if (F == E && j != k) s_bad = 1;  // duplicate page id
      rank += (s_pr[j] > pr) || (s_pr[j] == pr && F < E);
    }
    s_order[rank] = E;
  }
  __syncthreads();
  // Every check above has run (NaN fill scores, page spans, pending ids,
  // duplicates): a failed one ends the trajectory here, before any page span
  // is used to index the class bytes or a duplicate leaves a rank unwritten.
  if (s_bad) {
    if (threadIdx.x == 0) {
      record_error(hdr, COMMITKV_ERR_DEVICE_INPUT, -5);
      L.n_idx[t] = 0;
    }
    return;
  }
  if (threadIdx.x == 0) {
    // live entries occupy ranks [0, n_live); take the longest prefix that
    // fits both the page cap and the token budget B_N (Eq. 12)
    int n_live = 0;
    for (int k = 0; k < np; ++k) n_live += s_pid[k] >= 0;
    int pages = 0, toks = 0;
    for (int k = 0; k < n_live; ++k) s_take[k] = 0;
    for (int k = 0; k < n_live; ++k) {
      int E = s_order[k];
      int len = tr.pl[E];
      if (pages + 1 > L.cap || toks + len > L.B_N) break;
      s_take[k] = 1;
      ++pages;
      toks += len;
    }
    s_prot_tokens = toks;
    s_rem = n_live;  // reuse: number of ranked entries
  }
  __syncthreads();
  int n_live = s_rem;
  for (int k = 0; k < n_live; ++k) {
    if (!s_take[k]) break;
    int E = s_order[k];
    for (int i = tr.ps[E] + threadIdx.x; i < tr.ps[E] + tr.pl[E]; i += kThreads) cls[i] = 2;
  }
  __syncthreads();
  // fill: other non-retired tokens by (score desc, index desc) within the room
  int rem_local = 0;
  for (int i = threadIdx.x; i < S; i += kThreads) rem_local += cls[i] == 0;
  if (threadIdx.x == 0) s_rem = 0;
  __syncthreads();
  atomicAdd(&s_rem, rem_local);
  __syncthreads();
  int rem = s_rem;
  int room = L.B - s_prot_tokens;
  if (rem > room) {
    // exact k-th largest key (k = room) by 8-bit MSB-first radix select
    if (threadIdx.x == 0) {
      s_prefix = 0ull;
      s_krem = room;
      s_exact = 0;
    }
    unsigned long long mask = 0ull;
    // stops early once every key with the chosen prefix is taken: the
    // prefix (lower bits zero) is then itself the threshold
    for (int shift = 56; shift >= 0 && room > 0; shift -= 8) {
      for (int d = threadIdx.x; d < 256; d += kThreads) s_hist[d] = 0;
      __syncthreads();
      unsigned long long prefix = s_prefix;
      for (int i = threadIdx.x; i < S; i += kThreads) {
        if (cls[i] != 0) continue;
        uint64_t key = fill_key(L.fill[t][i], i);
        if ((key & mask) == prefix) atomicAdd(&s_hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x < 32) {
        // the first bin, from the top, at which the count of larger keys
        // reaches `need`: lane l holds bins 255 - 8 l down to 248 - 8 l, a
        // warp scan gives each lane the count above its bins, and the lane
        // whose bins hold the crossing walks them in order
        const int lane = threadIdx.x, need = s_krem;
        unsigned sum = 0;
#pragma unroll
        for (int u = 0; u < 8; ++u) sum += s_hist[255 - 8 * lane - u];
        unsigned incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, incl >= (unsigned)need);
        if (hit != 0u && lane == __ffs(hit) - 1) {
          unsigned cum = incl - sum;
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const unsigned c = s_hist[255 - 8 * lane - u];
            if (cum + c >= (unsigned)need) {
              s_prefix = prefix | ((unsigned long long)(255 - 8 * lane - u) << shift);
              s_krem = need - (int)cum;
              s_exact = s_krem == (int)c;
              break;
            }
            cum += c;
          }
        }
      }
      mask |= 255ull << shift;
      __syncthreads();
      if (s_exact) break;
    }
    unsigned long long thr = s_prefix;
    for (int i = threadIdx.x; i < S; i += kThreads)
      if (cls[i] == 0 && (room > 0 && fill_key(L.fill[t][i], i) >= thr)) cls[i] = 3;
  } else {
    for (int i = threadIdx.x; i < S; i += kThreads)
      if (cls[i] == 0) cls[i] = 3;
  }
  __syncthreads();
  // I_j ascending: protected (2) and kept (3) tokens; each thread takes a
  // contiguous segment, one block scan places the segments
  const int seg = (S + kThreads - 1) / kThreads;
  const int i0 = min(S, (int)threadIdx.x * seg), i1 = min(S, i0 + seg);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += cls[i] >= 2;
  int excl;
  const int total = block_scan(cnt, &excl, s_warp);
  for (int i = i0, o = excl; i < i1 && o < L.B; ++i)
    if (cls[i] >= 2) L.idx[t][o++] = i;
  if (threadIdx.x == 0) L.n_idx[t] = total < L.B ? total : L.B;
}

template <int VEC_BYTES>
__global__ void __launch_bounds__(256) gather_kernel(const __grid_constant__ CompactLaunch L) {
  int t = blockIdx.z;
  const TrajDev &tr = L.t[t];
  int slice = blockIdx.y;  // l * H + h
  int l = slice / L.H, h = slice % L.H;
  int row_bytes = L.d * L.elem_bytes;
  int vec_per_row = row_bytes / VEC_BYTES;
  int n = L.n_idx[t];
  int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int j = (int)(g / vec_per_row), vv = (int)(g % vec_per_row);
  if (j >= n) return;
  int i = L.idx[t][j];
  const char *ks = static_cast<const char *>(tr.k) + ((int64_t)l * tr.sl + (int64_t)h * tr.sh + (int64_t)i * tr.st) * L.elem_bytes;
  const char *vs = static_cast<const char *>(tr.v) + ((int64_t)l * tr.sl + (int64_t)h * tr.sh + (int64_t)i * tr.st) * L.elem_bytes;
  int64_t doff = (((int64_t)slice * L.B) + j) * row_bytes + (int64_t)vv * VEC_BYTES;
  if (L.k_out[t]) {
    if (VEC_BYTES == 16)
      *reinterpret_cast<uint4 *>(static_cast<char *>(L.k_out[t]) + doff) =
          *reinterpret_cast<const uint4 *>(ks + vv * VEC_BYTES);
    else
      *reinterpret_cast<uint16_t *>(static_cast<char *>(L.k_out[t]) + doff) =
          *reinterpret_cast<const uint16_t *>(ks + vv * VEC_BYTES);
  }
  if (L.v_out[t]) {
    if (VEC_BYTES == 16)
      *reinterpret_cast<uint4 *>(static_cast<char *>(L.v_out[t]) + doff) =
          *reinterpret_cast<const uint4 *>(vs + vv * VEC_BYTES);
    else
      *reinterpret_cast<uint16_t *>(static_cast<char *>(L.v_out[t]) + doff) =
          *reinterpret_cast<const uint16_t *>(vs + vv * VEC_BYTES);
  }
  if (slice == 0 && vv == 0 && L.pos_out[t]) L.pos_out[t][j] = tr.pos[i];
}

// In-place gather: one block per (K or V, layer, KV head, trajectory)
// slice.  I is strictly increasing with I_j >= j, so row j's destination is
// a source only for rows k <= j.  The block walks the slice in chunks of
// ROWS rows: it reads every source row of the chunk, waits at the barrier,
// then writes the chunk's destinations.  A destination in chunk c is read,
// if at all, by a row of chunk c or earlier, before that chunk's barrier;
// sources of later chunks lie at or after their own rows, past every row
// written so far.  Rows with I_j = j are left alone.
template <int VEC_BYTES, int ROWS>
__global__ void __launch_bounds__(256) gather_in_place_kernel(const __grid_constant__ CompactLaunch L) {
  using Vec = typename std::conditional<VEC_BYTES == 16, uint4, uint16_t>::type;
  constexpr int kMaxVec = 512 / VEC_BYTES;  // vectors per row at most (fp32, d = 128)
  constexpr int kPer = ROWS * kMaxVec / 256;
  const int t = blockIdx.z, slice = blockIdx.y;
  const TrajDev &tr = L.t[t];
  const int l = slice / L.H, h = slice % L.H;
  const int vpr = L.d * L.elem_bytes / VEC_BYTES;
  char *base = static_cast<char *>(const_cast<void *>(blockIdx.x ? tr.v : tr.k)) +
               ((int64_t)l * tr.sl + (int64_t)h * tr.sh) * L.elem_bytes;
  const int64_t rs = tr.st * L.elem_bytes;
  const int n = L.n_idx[t];
  const int32_t *idx = L.idx[t];
  for (int j0 = 0; j0 < n; j0 += ROWS) {
    Vec buf[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int e = threadIdx.x + 256 * u, r = e / vpr, w = e % vpr;
      if (r < ROWS && j0 + r < n) {
        const int i = idx[j0 + r];
        if (i != j0 + r) buf[u] = *reinterpret_cast<const Vec *>(base + i * rs + w * VEC_BYTES);
      }
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int e = threadIdx.x + 256 * u, r = e / vpr, w = e % vpr;
      if (r < ROWS && j0 + r < n) {
        const int i = idx[j0 + r];
        if (i != j0 + r) *reinterpret_cast<Vec *>(base + (int64_t)(j0 + r) * rs + w * VEC_BYTES) = buf[u];
      }
    }
  }
}

// Positions in place, one block per trajectory, by the same chunk rule.
__global__ void __launch_bounds__(256) positions_in_place_kernel(const __grid_constant__ CompactLaunch L) {
  const int t = blockIdx.x;
  int32_t *pos = const_cast<int32_t *>(L.t[t].pos);
  const int n = L.n_idx[t];
  const int32_t *idx = L.idx[t];
  for (int j0 = 0; j0 < n; j0 += 256) {
    const int j = j0 + threadIdx.x;
    int v = 0;
    if (j < n) v = pos[idx[j]];
    __syncthreads();
    if (j < n) pos[j] = v;
  }
}

}  // namespace

cudaError_t launch_compact(const CompactLaunch &L, WsHeader *hdr, cudaStream_t stream) {
  if (L.n_traj <= 0) return cudaSuccess;
  select_kernel<<<L.n_traj, kThreads, 0, stream>>>(L, hdr);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (L.in_place) {
    bool aligned = (L.d * L.elem_bytes) % 16 == 0;
    for (int t = 0; t < L.n_traj; ++t) {
      const TrajDev &tr = L.t[t];
      aligned &= ((uintptr_t)tr.k % 16 == 0) && ((uintptr_t)tr.v % 16 == 0) &&
                 ((tr.sl * L.elem_bytes) % 16 == 0) && ((tr.sh * L.elem_bytes) % 16 == 0) &&
                 ((tr.st * L.elem_bytes) % 16 == 0);
    }
    if (L.B == 0) return cudaSuccess;
    dim3 grid(2, L.M * L.H, L.n_traj);
    if (aligned) gather_in_place_kernel<16, 64><<<grid, 256, 0, stream>>>(L);
    else gather_in_place_kernel<2, 8><<<grid, 256, 0, stream>>>(L);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    positions_in_place_kernel<<<L.n_traj, 256, 0, stream>>>(L);
    return cudaGetLastError();
  }
  bool any_out = false;
  bool aligned = (L.d * L.elem_bytes) % 16 == 0;
  for (int t = 0; t < L.n_traj; ++t) {
    any_out |= L.k_out[t] || L.v_out[t] || L.pos_out[t];
    const TrajDev &tr = L.t[t];
    aligned &= ((uintptr_t)tr.k % 16 == 0) && ((uintptr_t)tr.v % 16 == 0) &&
               ((tr.sl * L.elem_bytes) % 16 == 0) && ((tr.sh * L.elem_bytes) % 16 == 0) &&
               ((tr.st * L.elem_bytes) % 16 == 0) &&
               ((uintptr_t)L.k_out[t] % 16 == 0) && ((uintptr_t)L.v_out[t] % 16 == 0);
  }
  if (!any_out || L.B == 0) return cudaSuccess;
  int row_bytes = L.d * L.elem_bytes;
  if (aligned) {
    int64_t threads = (int64_t)L.B * (row_bytes / 16);
    dim3 grid((unsigned)((threads + 255) / 256), L.M * L.H, L.n_traj);
    gather_kernel<16><<<grid, 256, 0, stream>>>(L);
  } else {
    int64_t threads = (int64_t)L.B * (row_bytes / 2);
    dim3 grid((unsigned)((threads + 255) / 256), L.M * L.H, L.n_traj);
    gather_kernel<2><<<grid, 256, 0, stream>>>(L);
  }
  return cudaGetLastError();
}

int compact_max_pending() { return kMaxPending; }

}  // namespace ckv
