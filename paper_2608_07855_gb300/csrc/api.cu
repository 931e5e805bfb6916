// C ABI of the CommitKV hot path: argument checks, workspace layout and
// launch sequences.  Every entry point is declared in include/commitkv.h.
#include <math.h>
#include <string.h>

#include <stdlib.h>

#include "ckv_internal.cuh"
#include "score_tc.cuh"

namespace ckv {
namespace ts {
cudaError_t launch_tc(const Batch &b, const float *const *stats, float *const *score, WsHeader *hdr,
                      cudaStream_t s, int sm_count);
cudaError_t launch_simt(const Batch &b, const float *const *stats, float *const *score, cudaStream_t s);
}  // namespace ts
int simt_rows_per_block();
int simt_pages_per_block();
int compact_max_pending();

commitkv_status check_shape(const commitkv_shape *s) {
  if (!s) return COMMITKV_ERR_INVALID_ARG;
  if (s->layers < 1 || s->layers > kMaxLayers || s->kv_heads < 1 || s->q_heads < s->kv_heads ||
      s->q_heads % s->kv_heads != 0 || s->head_dim < 1)
    return COMMITKV_ERR_INVALID_ARG;
  if (s->dtype != COMMITKV_F32 && s->dtype != COMMITKV_BF16) return COMMITKV_ERR_INVALID_ARG;
  if (!(s->softmax_scale >= 0.0f) || isinf(s->softmax_scale)) return COMMITKV_ERR_INVALID_ARG;
  if (s->head_dim != 64 && s->head_dim != 128) return COMMITKV_ERR_UNSUPPORTED;
  if ((int64_t)s->layers * s->q_heads > (1 << 20)) return COMMITKV_ERR_INVALID_ARG;
  return COMMITKV_OK;
}

commitkv_status check_trajs(const commitkv_shape *s, int n_traj, const commitkv_traj *tr,
                            bool need_q) {
  if (n_traj < 1 || n_traj > kMaxTraj || !tr) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t) {
    const commitkv_traj &x = tr[t];
    if (x.S < 0 || x.W < 0 || x.P < 0) return COMMITKV_ERR_INVALID_ARG;
    if (x.S > 0 && (!x.k || !x.v || !x.pos)) return COMMITKV_ERR_INVALID_ARG;
    if (x.P > 0 && (!x.page_start || !x.page_len)) return COMMITKV_ERR_INVALID_ARG;
    if (need_q && x.W > 0 && (!x.q || !x.q_pos)) return COMMITKV_ERR_INVALID_ARG;
    if (x.stride_tok < s->head_dim || x.stride_head < 0 || x.stride_layer < 0)
      return COMMITKV_ERR_INVALID_ARG;
    if ((int64_t)(s->q_heads / s->kv_heads) * x.W > (1 << 24)) return COMMITKV_ERR_INVALID_ARG;
  }
  return COMMITKV_OK;
}

// Host-side checks of the compression checkpoint's arguments, shared by
// commitkv_compact, commitkv_compact_in_place and commitkv_compact_noalloc.
commitkv_status check_compact_args(const commitkv_shape *s, int32_t n_traj, const commitkv_traj *tr,
                                   const uint8_t *const *retired, const int32_t *const *pending,
                                   const int32_t *n_pending, const float *const *pending_priority,
                                   const float *const *fill_score, int32_t budget_B,
                                   int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                   int32_t *const *idx_out, const int32_t *n_idx_out) {
  commitkv_status st = check_shape(s);
  if (st) return st;
  if ((st = check_trajs(s, n_traj, tr, false))) return st;
  if (budget_B < 0 || pending_tokens_BN < 0 || pending_tokens_BN > budget_B || pending_cap_pages < 0)
    return COMMITKV_ERR_INVALID_ARG;
  if (!retired || !n_pending || !fill_score || !idx_out || !n_idx_out) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t) {
    if (n_pending[t] < 0 || n_pending[t] > compact_max_pending()) return COMMITKV_ERR_INVALID_ARG;
    if (n_pending[t] > 0 && (!pending || !pending[t] || !pending_priority || !pending_priority[t]))
      return COMMITKV_ERR_INVALID_ARG;
    if (tr[t].P > 0 && !retired[t]) return COMMITKV_ERR_INVALID_ARG;
    if (tr[t].S > 0 && !fill_score[t]) return COMMITKV_ERR_INVALID_ARG;
    if (budget_B > 0 && !idx_out[t]) return COMMITKV_ERR_INVALID_ARG;
  }
  return COMMITKV_OK;
}

}  // namespace ckv

using namespace ckv;

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

int layers_selected(const commitkv_shape *s, const uint8_t *mask, uint8_t *ids) {
  int n = 0;
  for (int l = 0; l < s->layers; ++l)
    if (!mask || mask[l]) ids[n++] = (uint8_t)l;
  return n;
}

TrajDev to_dev(const commitkv_traj &x) {
  TrajDev d;
  d.k = x.k;
  d.v = x.v;
  d.sl = x.stride_layer;
  d.sh = x.stride_head;
  d.st = x.stride_tok;
  d.pos = x.pos;
  d.q = x.q;
  d.qpos = x.q_pos;
  d.ps = x.page_start;
  d.pl = x.page_len;
  d.S = x.S;
  d.W = x.W;
  d.P = x.P;
  d.pad = 0;
  return d;
}

void fill_batch(Batch &b, const commitkv_shape *s, int n_traj, const commitkv_traj *tr,
                const uint8_t *mask) {
  memset(&b, 0, sizeof b);
  b.n_traj = n_traj;
  b.M = s->layers;
  b.H = s->kv_heads;
  b.Hq = s->q_heads;
  b.g = s->q_heads / s->kv_heads;
  b.d = s->head_dim;
  b.dtype = s->dtype;
  b.scale = s->softmax_scale > 0.0f ? s->softmax_scale : 1.0f / sqrtf((float)s->head_dim);
  b.scale_log2 = b.scale * 1.4426950408889634f;
  b.n_layers = layers_selected(s, mask, b.layer_ids);
  for (int t = 0; t < n_traj; ++t) b.t[t] = to_dev(tr[t]);
}

int chunk_len_for(int n_traj, const commitkv_traj *tr) {
  int smax = 0;
  for (int t = 0; t < n_traj; ++t) smax = tr[t].S > smax ? tr[t].S : smax;
  int c = (smax + 15) / 16;
  if (c < 512) c = 512;
  return (c + 63) / 64 * 64;
}

int cdiv(int a, int b) { return (a + b - 1) / b; }

// ---- tensor-core scoring path (bf16, head_dim 128)
int tc_chunk_len(int n_traj, const commitkv_traj *tr) {
  int smax = 0;
  for (int t = 0; t < n_traj; ++t) smax = tr[t].S > smax ? tr[t].S : smax;
  int c = (smax + 7) / 8;  // at most 8 chunks per (layer, KV head)
  if (c < 1024) c = 1024;
  return (c + 127) / 128 * 128;
}

struct TcCounts {
  int nchunk, nrt, nbitem;
};

TcCounts tc_counts(const commitkv_shape *s, const commitkv_traj &x, int CL) {
  TcCounts c;
  int g = s->q_heads / s->kv_heads;
  c.nchunk = cdiv(x.S, CL);
  c.nrt = cdiv(g * x.W, tc::kRowsPerTile);
  c.nbitem = cdiv(cdiv(x.S, 16) + x.P, tc::kSlotsPerItem);
  return c;
}

bool env_force_simt() {
  const char *e = getenv("COMMITKV_SCORING");
  return e && (e[0] == 's' || e[0] == 'S');
}

bool tc_eligible(const commitkv_shape *s, int n_traj, const commitkv_traj *tr) {
  if (s->dtype != COMMITKV_BF16 || s->head_dim != 128 || env_force_simt()) return false;
  for (int t = 0; t < n_traj; ++t) {
    const commitkv_traj &x = tr[t];
    if (x.S == 0 || x.W == 0 || x.P == 0) continue;
    if (((uintptr_t)x.k | (uintptr_t)x.v | (uintptr_t)x.q) % 16) return false;
    if ((x.stride_tok * 2) % 16 || (x.stride_head * 2) % 16 || (x.stride_layer * 2) % 16) return false;
    if (x.stride_head == 0 || x.stride_layer == 0) return false;
  }
  return true;
}

// Chunks per (layer, KV head) never exceed 16 nor ceil(S / 1024) for the
// tensor-core path (ceil(S / 512) for the CUDA-core path), whatever S' <= S a
// later call uses: the workspace bound below holds for smaller caches too.
int tc_chunk_bound(int S) {
  int c = cdiv(S, 1024);
  return c < 16 ? c : 16;
}
int simt_chunk_bound(int S) {
  int c = cdiv(S, 512);
  return c < 16 ? c : 16;
}

// The single cooperative launch of both scoring passes is opt-in
// (COMMITKV_FUSED=1): both passes are bound by their SMs' pipelines rather
// than by HBM, so serving the page pass's re-reads from L2 does not make it
// faster, and the fused launch measured slower than the separate launches.
bool env_fused() {
  const char *e = getenv("COMMITKV_FUSED");
  return e && e[0] == '1';
}

// Flash-pass partial slots the tensor-core path may need for these caches or
// smaller ones: one per item of the two-launch chunking, or the fused
// launch's ring (at most kMaxFusedCtas x kPartialRing slots, and at most one
// per item of its chunking: about kFusedItemsPerSlice items per slice).
size_t tc_partial_slots(const commitkv_shape *s, int n_traj, const commitkv_traj *tr) {
  size_t items = 0, fused = 0;
  for (int t = 0; t < n_traj; ++t) {
    TcCounts c = tc_counts(s, tr[t], tc_chunk_len(1, &tr[t]));
    items += (size_t)s->layers * s->kv_heads * tc_chunk_bound(tr[t].S) * c.nrt;
    fused += (size_t)s->layers * s->kv_heads * (tc::kFusedItemsPerSlice + 1 + c.nrt);
  }
  const size_t ring = (size_t)tc::kMaxFusedCtas * tc::kPartialRing;
  if (fused > ring) fused = ring;
  return items > fused ? items : fused;
}

size_t tc_score_bytes(const commitkv_shape *s, int n_traj, const commitkv_traj *tr) {
  size_t slots = 0, slices = 0;
  for (int t = 0; t < n_traj; ++t) {
    TcCounts c = tc_counts(s, tr[t], tc_chunk_len(1, &tr[t]));
    slots += align_up((size_t)(tr[t].P + 1) * 4) + align_up((size_t)c.nbitem * 32) + kAlign +
             align_up(((size_t)cdiv(tr[t].S, 16) + tr[t].P) * 16);
    slices += (size_t)s->layers * s->kv_heads;
  }
  return align_up(tc_partial_slots(s, n_traj, tr) * tc::kPartsPerItem * tc::kRowsPerTile * 132 * 4) +
         align_up(slices * 2 * tc::kCounterStride * 4) + slots;
}

// Region sizes of each call (bytes after the 256-byte header).
size_t score_bytes(const commitkv_shape *s, int n_traj, const commitkv_traj *tr, int n_layers) {
  int CL = chunk_len_for(n_traj, tr), RB = simt_rows_per_block(), d = s->head_dim;
  int g = s->q_heads / s->kv_heads;
  size_t units = 0, stats = 0;
  (void)CL;
  for (int t = 0; t < n_traj; ++t) {
    int rows = g * tr[t].W;
    units += (size_t)n_layers * s->kv_heads * simt_chunk_bound(tr[t].S) * cdiv(rows, RB);
    stats += align_up((size_t)s->layers * s->q_heads * tr[t].W * (d + 4) * 4) + align_up((size_t)tr[t].W * 4);
  }
  size_t scratch = align_up(units * RB * (d + 4) * 4);
  if (s->head_dim == 128) {
    size_t tcb = tc_score_bytes(s, n_traj, tr);
    if (tcb > scratch) scratch = tcb;
  }
  return scratch + stats;
}

size_t joint_bytes(const commitkv_shape *s, int n_traj, const commitkv_traj *tr, int n_layers) {
  int g = s->q_heads / s->kv_heads, d = s->head_dim, k = joint_round();
  size_t rows = 0;
  for (int t = 0; t < n_traj; ++t) rows += (size_t)n_layers * s->kv_heads * g * tr[t].W;
  return align_up(rows * d * 4) + align_up((size_t)k * rows * d * 4) + align_up(rows * 8) +
         align_up((size_t)k * rows * 8) + align_up((size_t)3 * n_traj * joint_combos() * 4);
}

size_t classify_bytes(int n_traj, const int32_t *P) {
  size_t b = 0;
  for (int t = 0; t < n_traj; ++t) b += align_up((size_t)P[t] * 4);
  return b;
}

size_t compact_bytes(int n_traj, const commitkv_traj *tr) {
  size_t b = 0;
  for (int t = 0; t < n_traj; ++t) b += align_up((size_t)tr[t].S);
  return b;
}

commitkv_status check_ws(void *ws, size_t bytes, size_t need) {
  if (!ws || ((uintptr_t)ws % kAlign) != 0) return COMMITKV_ERR_WORKSPACE;
  if (bytes < need) return COMMITKV_ERR_WORKSPACE;
  return COMMITKV_OK;
}

commitkv_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return COMMITKV_OK;
  cudaGetLastError();  // clear the sticky-free error state of this thread
  return COMMITKV_ERR_CUDA;
}

}  // namespace

extern "C" {

size_t commitkv_workspace_size(const commitkv_shape *shape, int32_t n_traj,
                               const commitkv_traj *trajs) {
  if (check_shape(shape) != COMMITKV_OK) return 0;
  if (check_trajs(shape, n_traj, trajs, false) != COMMITKV_OK) return 0;
  int32_t P[kMaxTraj];
  for (int t = 0; t < n_traj; ++t) P[t] = trajs[t].P;
  size_t need = score_bytes(shape, n_traj, trajs, shape->layers);
  size_t j = joint_bytes(shape, n_traj, trajs, shape->layers);
  size_t c = classify_bytes(n_traj, P);
  size_t k = compact_bytes(n_traj, trajs);
  if (j > need) need = j;
  if (c > need) need = c;
  if (k > need) need = k;
  return kAlign + need;
}

commitkv_status commitkv_workspace_init(void *workspace, size_t workspace_bytes,
                                        cudaStream_t stream) {
  if (!workspace || workspace_bytes < kAlign || ((uintptr_t)workspace % kAlign)) return COMMITKV_ERR_WORKSPACE;
  return cuda_status(cudaMemsetAsync(workspace, 0, sizeof(WsHeader), stream));
}

commitkv_status commitkv_workspace_status(const void *workspace, size_t workspace_bytes,
                                          cudaStream_t stream, int32_t clear) {
  if (!workspace || workspace_bytes < kAlign || ((uintptr_t)workspace % kAlign)) return COMMITKV_ERR_WORKSPACE;
  WsHeader h;
  cudaError_t e = cudaMemcpyAsync(&h, workspace, sizeof h, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_status(e);
  if (clear) {
    e = cudaMemsetAsync(const_cast<void *>(workspace), 0, sizeof(WsHeader), stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return (commitkv_status)h.status;
}

const char *commitkv_status_string(commitkv_status s) {
  switch (s) {
    case COMMITKV_OK: return "ok";
    case COMMITKV_ERR_INVALID_ARG: return "invalid argument";
    case COMMITKV_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case COMMITKV_ERR_CUDA: return "CUDA runtime error";
    case COMMITKV_ERR_TIMEOUT: return "bounded device wait timed out";
    case COMMITKV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case COMMITKV_ERR_DEVICE_INPUT: return "device-resident input failed a device-side check";
  }
  return "unknown status";
}

namespace {

// Scoring of both entry points: with stats_in the row stats are the
// caller's and only the page pass runs.
commitkv_status page_effects_impl(const commitkv_shape *shape, int32_t n_traj, const commitkv_traj *trajs,
                                  const uint8_t *layer_mask, const float *const *stats_in,
                                  float *const *R_out, float *const *head_R_out, float *const *stats_out,
                                  void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  commitkv_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_trajs(shape, n_traj, trajs, true))) return st;
  if (!R_out) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t) {
    if (trajs[t].P > 0 && !R_out[t]) return COMMITKV_ERR_INVALID_ARG;
    if (stats_in && trajs[t].P > 0 && trajs[t].W > 0 && !stats_in[t]) return COMMITKV_ERR_INVALID_ARG;
  }
  const bool from_stats = stats_in != nullptr;

  static thread_local ScoreLaunch L;  // large: keep off the stack
  memset(&L, 0, sizeof L);
  fill_batch(L.batch, shape, n_traj, trajs, layer_mask);
  int nl = L.batch.n_layers;
  size_t need = kAlign + score_bytes(shape, n_traj, trajs, shape->layers);
  if ((st = check_ws(workspace, workspace_bytes, need))) return st;

  int CL = chunk_len_for(n_traj, trajs), RB = simt_rows_per_block(), PG = simt_pages_per_block();
  int g = L.batch.g, d = shape->head_dim;
  L.chunk_len = CL;
  char *base = static_cast<char *>(workspace) + kAlign;
  size_t units = 0;
  for (int t = 0; t < n_traj; ++t) {
    int rows = g * trajs[t].W;
    L.nrb[t] = cdiv(rows, RB);
    L.nchunk[t] = cdiv(trajs[t].S, CL);
    L.npg[t] = cdiv(trajs[t].P, PG);
    L.unit_off_a[t + 1] = L.unit_off_a[t] + nl * shape->kv_heads * L.nchunk[t] * L.nrb[t];
    L.unit_off_b[t + 1] = L.unit_off_b[t] + nl * shape->kv_heads * L.npg[t] * L.nrb[t];
    L.row_off[t + 1] = L.row_off[t] + nl * shape->kv_heads * rows;
    units += (size_t)nl * shape->kv_heads * L.nchunk[t] * L.nrb[t];
  }
  float *partials = reinterpret_cast<float *>(base);
  // scratch (either path's partials) first, then the stats of trajectories
  // without stats_out; the layout is computed for every layer
  size_t full_units = 0;
  for (int t = 0; t < n_traj; ++t)
    full_units += (size_t)shape->layers * shape->kv_heads * simt_chunk_bound(trajs[t].S) * L.nrb[t];
  size_t scratch = align_up(full_units * RB * (d + 4) * 4);
  if (shape->head_dim == 128) {
    size_t tcb = tc_score_bytes(shape, n_traj, trajs);
    if (tcb > scratch) scratch = tcb;
  }
  char *sbase = base + scratch;
  for (int t = 0; t < n_traj; ++t) {
    size_t sb = align_up((size_t)shape->layers * shape->q_heads * trajs[t].W * (d + 4) * 4);
    if (from_stats) L.stats[t] = const_cast<float *>(stats_in[t]);  // read only
    else L.stats[t] = (stats_out && stats_out[t]) ? stats_out[t] : reinterpret_cast<float *>(sbase);
    sbase += sb;
    L.R[t] = R_out[t];
    L.headR[t] = head_R_out ? head_R_out[t] : nullptr;
  }
  for (int t = 0; t < n_traj; ++t) {
    L.nvis_w[t] = reinterpret_cast<int32_t *>(sbase);
    sbase += align_up((size_t)trajs[t].W * 4);
  }
  L.from_stats = from_stats ? 1 : 0;
  for (int t = 0; t < n_traj; ++t) {
    if (trajs[t].P == 0) continue;
    cudaError_t e = cudaMemsetAsync(R_out[t], 0, (size_t)trajs[t].P * 4, stream);
    if (e == cudaSuccess && L.headR[t])
      e = cudaMemsetAsync(L.headR[t], 0, (size_t)shape->layers * shape->q_heads * trajs[t].P * 4, stream);
    if (e != cudaSuccess) return cuda_status(e);
  }
  WsHeader *hdr = static_cast<WsHeader *>(workspace);
  if (!tc_eligible(shape, n_traj, trajs)) return cuda_status(launch_score_simt(L, partials, hdr, stream));
  // tensor-core path: trajectories in launches of up to tc::kMaxTc
  static thread_local tc::TcLaunch T;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_status(e);
  const bool fused = !from_stats && env_fused();
  int CLt = tc_chunk_len(n_traj, trajs);
  if (fused) {
    int smax = 0, nrt_max = 1;
    for (int t = 0; t < n_traj; ++t) {
      smax = trajs[t].S > smax ? trajs[t].S : smax;
      const int nrt = cdiv(L.batch.g * trajs[t].W, tc::kRowsPerTile);
      nrt_max = nrt > nrt_max ? nrt : nrt_max;
    }
    CLt = tc::fused_chunk_len(smax, nrt_max);
  }
  float *tc_partials = reinterpret_cast<float *>(base);
  size_t slices_all = 0;
  for (int t = 0; t < n_traj; ++t) slices_all += (size_t)shape->layers * shape->kv_heads;
  char *cnt_base = base + align_up(tc_partial_slots(shape, n_traj, trajs) * tc::kPartsPerItem * tc::kRowsPerTile *
                                   132 * 4);
  char *slot_base = cnt_base + align_up(slices_all * 2 * tc::kCounterStride * 4);
  for (int b0 = 0; b0 < n_traj; b0 += tc::kMaxTc) {
    int nb = n_traj - b0 < tc::kMaxTc ? n_traj - b0 : tc::kMaxTc;
    memset(&T, 0, sizeof T);
    T.n_traj = nb;
    T.M = shape->layers;
    T.H = shape->kv_heads;
    T.Hq = shape->q_heads;
    T.g = L.batch.g;
    T.n_layers = nl;
    T.chunk_len = CLt;
    T.slots_per_item = tc::kSlotsPerItem;
    T.from_stats = L.from_stats;
    T.scale_log2 = L.batch.scale_log2;
    T.partials = tc_partials;
    T.fused = fused ? 1 : 0;
    T.a_done = reinterpret_cast<uint32_t *>(cnt_base);
    T.merged = T.a_done + slices_all * tc::kCounterStride;
    memcpy(T.layer_ids, L.batch.layer_ids, sizeof T.layer_ids);
    for (int i = 0; i < nb; ++i) {
      int t = b0 + i;
      const commitkv_traj &x = trajs[t];
      TcCounts c = tc_counts(shape, x, CLt);
      tc::TcTraj &tt = T.t[i];
      tt.pos = x.pos;
      tt.qpos = x.q_pos;
      tt.ps = x.page_start;
      tt.pl = x.page_len;
      tt.slot_off = reinterpret_cast<int32_t *>(slot_base);
      slot_base += align_up((size_t)(x.P + 1) * 4);
      tt.items = reinterpret_cast<int4 *>(slot_base);
      slot_base += align_up((size_t)c.nbitem * 32);
      tt.prep = reinterpret_cast<tc::TcPrep *>(slot_base);
      slot_base += kAlign;
      tt.slot_tab = reinterpret_cast<int4 *>(slot_base);
      slot_base += align_up(((size_t)cdiv(x.S, 16) + x.P) * 16);
      tt.stats = L.stats[t];
      tt.nvis_w = L.nvis_w[t];
      tt.R = L.R[t];
      tt.headR = L.headR[t];
      tt.S = x.S;
      tt.W = x.W;
      tt.P = x.P;
      tt.nchunk = c.nchunk;
      tt.nrt = c.nrt;
      tt.nbitem = c.nbitem;
      bool active = x.S > 0 && x.W > 0;
      int ia = active ? nl * shape->kv_heads * c.nchunk * c.nrt : 0;
      int ib = active && x.P > 0 ? nl * shape->kv_heads * c.nbitem * c.nrt : 0;
      T.item_off_a[i + 1] = T.item_off_a[i] + ia;
      T.item_off_b[i + 1] = T.item_off_b[i] + ib;
      T.row_off[i + 1] = T.row_off[i] + (active ? nl * shape->kv_heads * L.batch.g * x.W : 0);
      T.slice_off[i + 1] = T.slice_off[i] + (active ? nl * shape->kv_heads : 0);
      if (active && !tc::build_maps(T.maps[i], L.batch.t[t], shape->layers, shape->kv_heads, shape->q_heads))
        return COMMITKV_ERR_CUDA;
    }
    e = tc::launch_score_tc(T, hdr, stream, sms);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return COMMITKV_OK;
}

}  // namespace

commitkv_status commitkv_page_effects(const commitkv_shape *shape, int32_t n_traj,
                                      const commitkv_traj *trajs, const uint8_t *layer_mask,
                                      float *const *R_out, float *const *head_R_out,
                                      float *const *stats_out, void *workspace,
                                      size_t workspace_bytes, cudaStream_t stream) {
  return page_effects_impl(shape, n_traj, trajs, layer_mask, nullptr, R_out, head_R_out, stats_out, workspace,
                           workspace_bytes, stream);
}

commitkv_status commitkv_page_effects_from_stats(const commitkv_shape *shape, int32_t n_traj,
                                                 const commitkv_traj *trajs, const uint8_t *layer_mask,
                                                 const float *const *stats_in, float *const *R_out,
                                                 float *const *head_R_out, void *workspace,
                                                 size_t workspace_bytes, cudaStream_t stream) {
  if (!stats_in) return COMMITKV_ERR_INVALID_ARG;
  return page_effects_impl(shape, n_traj, trajs, layer_mask, stats_in, R_out, head_R_out, nullptr, workspace,
                           workspace_bytes, stream);
}

commitkv_status commitkv_token_scores(const commitkv_shape *shape, int32_t n_traj, const commitkv_traj *trajs,
                                      const uint8_t *layer_mask, const float *const *stats,
                                      float *const *scores_out, void *workspace, size_t workspace_bytes,
                                      cudaStream_t stream) {
  commitkv_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_trajs(shape, n_traj, trajs, true))) return st;
  if (!stats || !scores_out) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t) {
    if (trajs[t].S > 0 && !scores_out[t]) return COMMITKV_ERR_INVALID_ARG;
    if (trajs[t].S > 0 && trajs[t].W > 0 && !stats[t]) return COMMITKV_ERR_INVALID_ARG;
  }
  if ((st = check_ws(workspace, workspace_bytes, kAlign))) return st;
  static thread_local Batch B;
  fill_batch(B, shape, n_traj, trajs, layer_mask);
  for (int t = 0; t < n_traj; ++t) {
    if (trajs[t].S == 0) continue;
    cudaError_t e = cudaMemsetAsync(scores_out[t], 0, (size_t)trajs[t].S * 4, stream);
    if (e != cudaSuccess) return cuda_status(e);
  }
  if (B.n_layers == 0) return COMMITKV_OK;
  // tensor cores for bf16, head_dim 128 and 16-byte aligned rows
  bool tc = shape->dtype == COMMITKV_BF16 && shape->head_dim == 128 && !env_force_simt();
  for (int t = 0; t < n_traj && tc; ++t) {
    const commitkv_traj &x = trajs[t];
    if (x.S == 0 || x.W == 0) continue;
    if (((uintptr_t)x.k | (uintptr_t)x.q | (uintptr_t)stats[t]) % 16) tc = false;
    if ((x.stride_tok * 2) % 16 || (x.stride_head * 2) % 16 || (x.stride_layer * 2) % 16) tc = false;
    if (x.stride_head == 0 || x.stride_layer == 0) tc = false;
  }
  WsHeader *hdr = static_cast<WsHeader *>(workspace);
  if (!tc) return cuda_status(ts::launch_simt(B, stats, scores_out, stream));
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = ts::launch_tc(B, stats, scores_out, hdr, stream, sms);
  return cuda_status(e);
}

commitkv_status commitkv_classify(int32_t n_traj, const int32_t *P, const float *const *R_pre,
                                  const float *const *R_post, const uint8_t *const *eligible,
                                  const commitkv_thresholds *thresholds, uint8_t *const *state_out,
                                  int32_t *const *cand_out, int32_t *n_cand_out, void *workspace,
                                  size_t workspace_bytes, cudaStream_t stream) {
  return commitkv_classify_variant(n_traj, P, R_pre, R_post, eligible, thresholds, 0u, state_out, cand_out,
                                   n_cand_out, workspace, workspace_bytes, stream);
}

commitkv_status commitkv_classify_variant(int32_t n_traj, const int32_t *P, const float *const *R_pre,
                                          const float *const *R_post, const uint8_t *const *eligible,
                                          const commitkv_thresholds *thresholds, uint32_t variant,
                                          uint8_t *const *state_out, int32_t *const *cand_out,
                                          int32_t *n_cand_out, void *workspace, size_t workspace_bytes,
                                          cudaStream_t stream) {
  if (n_traj < 1 || n_traj > kMaxTraj || !P || !R_pre || !R_post || !eligible || !state_out ||
      !cand_out || !n_cand_out)
    return COMMITKV_ERR_INVALID_ARG;
  if (variant & ~(uint32_t)(COMMITKV_CLASSIFY_NO_PRECOMMIT | COMMITKV_CLASSIFY_NO_PERCENTILE))
    return COMMITKV_ERR_INVALID_ARG;
  commitkv_thresholds th = thresholds ? *thresholds : commitkv_thresholds{0.05f, 0.01f, 0.75f, 0.25f};
  if (!(th.tau_dead < th.tau_use) || !(th.rho_dead < th.rho_use)) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t) {
    if (P[t] < 0) return COMMITKV_ERR_INVALID_ARG;
    if (P[t] > 0 && (!R_pre[t] || !R_post[t] || !eligible[t] || !state_out[t] || !cand_out[t]))
      return COMMITKV_ERR_INVALID_ARG;
  }
  commitkv_status st = check_ws(workspace, workspace_bytes, kAlign + classify_bytes(n_traj, P));
  if (st) return st;
  ClassifyLaunch L;
  memset(&L, 0, sizeof L);
  L.n_traj = n_traj;
  char *base = static_cast<char *>(workspace) + kAlign;
  for (int t = 0; t < n_traj; ++t) {
    L.P[t] = P[t];
    L.Rm[t] = R_pre[t];
    L.Rp[t] = R_post[t];
    L.el[t] = eligible[t];
    L.state[t] = state_out[t];
    L.cand[t] = cand_out[t];
    L.scratch[t] = reinterpret_cast<int32_t *>(base);
    base += align_up((size_t)P[t] * 4);
  }
  L.n_cand = n_cand_out;
  L.tau_use = th.tau_use;
  L.tau_dead = th.tau_dead;
  L.rho_use = (double)th.rho_use;
  L.rho_dead = (double)th.rho_dead;
  L.variant = variant;
  return cuda_status(launch_classify(L, static_cast<WsHeader *>(workspace), stream));
}

commitkv_status commitkv_joint_test(const commitkv_shape *shape, int32_t n_traj,
                                    const commitkv_traj *post, const uint8_t *layer_mask,
                                    const float *const *stats, const int32_t *const *cand,
                                    const int32_t *n_cand, float tau_joint,
                                    uint8_t *const *accepted_out, float *const *step_R_out,
                                    void *workspace, size_t workspace_bytes,
                                    cudaStream_t stream) {
  commitkv_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_trajs(shape, n_traj, post, true))) return st;
  if (!stats || !cand || !n_cand || !accepted_out || isnan(tau_joint)) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj; ++t)
    if (post[t].P > 0 && (!stats[t] || !cand[t] || !accepted_out[t])) return COMMITKV_ERR_INVALID_ARG;
  size_t need = kAlign + joint_bytes(shape, n_traj, post, shape->layers);
  if ((st = check_ws(workspace, workspace_bytes, need))) return st;

  static thread_local JointLaunch L;
  memset(&L, 0, sizeof L);
  fill_batch(L.batch, shape, n_traj, post, layer_mask);
  for (int t = 0; t < n_traj; ++t) L.stats[t] = stats[t];
  int nl = L.batch.n_layers, g = L.batch.g, d = shape->head_dim, RB = joint_rows_per_group(L);
  size_t rows_total = 0;
  int maxP = 0;
  for (int t = 0; t < n_traj; ++t) {
    int rows = g * post[t].W;
    L.nrb[t] = cdiv(rows, RB);
    L.group_off[t + 1] = L.group_off[t] + nl * shape->kv_heads * L.nrb[t];
    L.row_off[t + 1] = L.row_off[t] + nl * shape->kv_heads * rows;
    rows_total += (size_t)nl * shape->kv_heads * rows;
    maxP = post[t].P > maxP ? post[t].P : maxP;
  }
  size_t rows_full = 0;
  for (int t = 0; t < n_traj; ++t) rows_full += (size_t)shape->layers * shape->kv_heads * g * post[t].W;
  const size_t K = (size_t)joint_round(), tab_bytes = (size_t)3 * n_traj * joint_combos() * 4;
  char *base = static_cast<char *>(workspace) + kAlign;
  L.DA = reinterpret_cast<float *>(base);
  base += align_up(rows_full * d * 4);
  L.DE = reinterpret_cast<float *>(base);
  base += align_up(K * rows_full * d * 4);
  L.SA = reinterpret_cast<float *>(base);
  base += align_up(rows_full * 8);
  L.SE = reinterpret_cast<float *>(base);
  base += align_up(K * rows_full * 8);
  L.roundR = reinterpret_cast<float *>(base);
  L.rows_full = (int64_t)rows_full;
  for (int t = 0; t < n_traj; ++t) {
    L.cand[t] = cand[t];
    L.accepted[t] = accepted_out[t];
    L.stepR_out[t] = step_R_out ? step_R_out[t] : nullptr;
  }
  L.n_cand = n_cand;
  L.tau = tau_joint;
  cudaError_t e = cudaMemsetAsync(L.DA, 0, rows_total * d * 4, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(L.SA, 0, rows_full * 8, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(L.roundR, 0, tab_bytes, stream);
  for (int t = 0; t < n_traj && e == cudaSuccess; ++t)
    if (post[t].P > 0) e = cudaMemsetAsync(accepted_out[t], 0, post[t].P, stream);
  // the barrier counters start from a known state
  WsHeader *hdr = static_cast<WsHeader *>(workspace);
  if (e == cudaSuccess) e = cudaMemsetAsync(&hdr->abort, 0, 3 * sizeof(int32_t), stream);
  if (e != cudaSuccess) return cuda_status(e);
  if (rows_total == 0 || maxP == 0) return COMMITKV_OK;
  int dev = 0, sms = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_status(e);
  return cuda_status(launch_joint(L, hdr, stream, sms));
}

static commitkv_status compact_impl(const commitkv_shape *shape, int32_t n_traj,
                                    const commitkv_traj *cache, const uint8_t *const *retired,
                                    const int32_t *const *pending, const int32_t *n_pending,
                                    const float *const *pending_priority,
                                    const float *const *fill_score, int32_t budget_B,
                                    int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                    int32_t *const *idx_out, int32_t *n_idx_out,
                                    void *const *k_out, void *const *v_out, int32_t *const *pos_out,
                                    void *workspace, size_t workspace_bytes, cudaStream_t stream,
                                    bool in_place) {
  commitkv_status st = check_compact_args(shape, n_traj, cache, retired, pending, n_pending, pending_priority,
                                          fill_score, budget_B, pending_tokens_BN, pending_cap_pages, idx_out,
                                          n_idx_out);
  if (st) return st;
  if ((st = check_ws(workspace, workspace_bytes, kAlign + compact_bytes(n_traj, cache)))) return st;
  static thread_local CompactLaunch L;
  memset(&L, 0, sizeof L);
  L.n_traj = n_traj;
  L.M = shape->layers;
  L.H = shape->kv_heads;
  L.d = shape->head_dim;
  L.elem_bytes = shape->dtype == COMMITKV_BF16 ? 2 : 4;
  char *base = static_cast<char *>(workspace) + kAlign;
  for (int t = 0; t < n_traj; ++t) {
    L.t[t] = to_dev(cache[t]);
    L.retired[t] = retired[t];
    L.pending[t] = n_pending[t] ? pending[t] : nullptr;
    L.n_pending[t] = n_pending[t];
    L.prio[t] = n_pending[t] ? pending_priority[t] : nullptr;
    L.fill[t] = fill_score[t];
    L.cls[t] = reinterpret_cast<uint8_t *>(base);
    base += align_up((size_t)cache[t].S);
    L.idx[t] = idx_out[t];
    L.k_out[t] = k_out ? k_out[t] : nullptr;
    L.v_out[t] = v_out ? v_out[t] : nullptr;
    L.pos_out[t] = pos_out ? pos_out[t] : nullptr;
  }
  L.n_idx = n_idx_out;
  L.B = budget_B;
  L.B_N = pending_tokens_BN;
  L.cap = pending_cap_pages;
  L.in_place = in_place ? 1 : 0;
  return cuda_status(launch_compact(L, static_cast<WsHeader *>(workspace), stream));
}

commitkv_status commitkv_compact(const commitkv_shape *shape, int32_t n_traj,
                                 const commitkv_traj *cache, const uint8_t *const *retired,
                                 const int32_t *const *pending, const int32_t *n_pending,
                                 const float *const *pending_priority,
                                 const float *const *fill_score, int32_t budget_B,
                                 int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                 int32_t *const *idx_out, int32_t *n_idx_out,
                                 void *const *k_out, void *const *v_out, int32_t *const *pos_out,
                                 void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  return compact_impl(shape, n_traj, cache, retired, pending, n_pending, pending_priority, fill_score, budget_B,
                      pending_tokens_BN, pending_cap_pages, idx_out, n_idx_out, k_out, v_out, pos_out, workspace,
                      workspace_bytes, stream, false);
}

commitkv_status commitkv_compact_in_place(const commitkv_shape *shape, int32_t n_traj,
                                          const commitkv_traj *cache, const uint8_t *const *retired,
                                          const int32_t *const *pending, const int32_t *n_pending,
                                          const float *const *pending_priority,
                                          const float *const *fill_score, int32_t budget_B,
                                          int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                          int32_t *const *idx_out, int32_t *n_idx_out, void *workspace,
                                          size_t workspace_bytes, cudaStream_t stream) {
  if (!cache) return COMMITKV_ERR_INVALID_ARG;
  for (int t = 0; t < n_traj && t < COMMITKV_MAX_TRAJ; ++t)
    if (cache[t].S > 0 && (!cache[t].k || !cache[t].v || !cache[t].pos)) return COMMITKV_ERR_INVALID_ARG;
  return compact_impl(shape, n_traj, cache, retired, pending, n_pending, pending_priority, fill_score, budget_B,
                      pending_tokens_BN, pending_cap_pages, idx_out, n_idx_out, nullptr, nullptr, nullptr,
                      workspace, workspace_bytes, stream, true);
}

}  // extern "C"
