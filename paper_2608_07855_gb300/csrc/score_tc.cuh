// Launch description of the tensor-core scoring path (score_tc.cu).
#pragma once

#include <cuda.h>

#include "ckv_internal.cuh"

namespace ckv {
namespace tc {

constexpr int kMaxTc = 16;          // trajectories per launch (tensor maps travel as parameters)
constexpr int kRowsPerTile = 128;   // probe rows per MMA tile
constexpr int kSlotsPerItem = 128;  // 16-token slots per pass-B work item
constexpr int kPartsPerItem = 1;    // pass-A partials per work item (the two softmax groups merged)
constexpr int kPartialRing = 4;     // partial slots (items) per flash CTA of the fused launch
constexpr int kMaxFusedCtas = 256;  // bound on the fused launch's flash CTAs (workspace sizing)
constexpr int kFusedItemsPerSlice = 32;    // flash items per slice in the fused launch (chunking target)
constexpr double kFusedFlashShare = 0.55;  // share of the SMs that run the flash pass in the fused launch
constexpr int kCounterStride = 32;  // per-slice counters of the fused launch, one 128-byte line each

struct TcMaps {
  CUtensorMap q;             // Q as [M*Hq*W rows][128], box 64 x 128
  CUtensorMap k, v;          // K, V as [M][H][S][128], box 64 x 128 x 1 x 1
  CUtensorMap kb[3], vb[3];  // the same with 16-, 32- and 64-row boxes (runs of page slots)
};

// Per-trajectory facts computed once per call by the prep kernel.
struct TcPrep {
  int vis_all;  // leading resident tokens visible to every probe row
  int pad[3];
};

struct TcTraj {
  const int32_t *pos, *qpos, *ps, *pl;
  int32_t *slot_off;  // workspace [P + 1]
  int4 *items;        // workspace [nbitem][2]: {E0, E1, slot0, nslot}, {npages, 0, 0, 0}
  int4 *slot_tab;     // workspace [ceil(S/16) + P]: {tok0, nv, page, first | last << 1 | rank << 2}
  TcPrep *prep;       // workspace
  int32_t *nvis_w;    // workspace [W]: resident tokens visible to each window position
  float *stats;       // [M][Hq][W][132]
  float *R;           // [P]
  float *headR;       // [M][Hq][P] or null
  int S, W, P, nchunk, nrt, nbitem;
};

struct TcLaunch {
  TcMaps maps[kMaxTc];
  TcTraj t[kMaxTc];
  int n_traj, M, H, Hq, g, n_layers, chunk_len, slots_per_item;
  int from_stats;  // the stats are the caller's: no flash pass, no combine
  float scale_log2;
  float *partials;  // [items_a or n_a * kPartialRing][2][128][132]: one partial per softmax warpgroup
  int item_off_a[kMaxTc + 1], item_off_b[kMaxTc + 1], row_off[kMaxTc + 1];
  // fused launch: CTAs [0, n_a) run the flash pass, the rest the page pass
  int fused;  // 1: one cooperative launch of both passes (set by the caller; needs !from_stats)
  int n_a;    // set by launch_score_tc
  int slice_off[kMaxTc + 1];  // (trajectory, selected layer, KV head) slices: prefix per trajectory
  uint32_t *a_done;           // workspace [slices][kCounterStride]: flash-pass warps done with their partials
  uint32_t *merged;           // workspace [slices][kCounterStride]: merge warps done with their rows
  uint8_t layer_ids[kMaxLayers];
};

size_t smem_a();
size_t smem_b();
bool build_maps(TcMaps &maps, const TrajDev &t, int M, int H, int Hq);
cudaError_t launch_score_tc(TcLaunch &L, WsHeader *hdr, cudaStream_t stream, int sm_count);
// Flash-pass CTAs of a fused launch on sm_count SMs (the rest run the page pass).
int fused_flash_ctas(const TcLaunch &L, int sm_count);
// Chunk length (tokens) of the fused launch for caches of up to max_tokens
// tokens and max_row_tiles 128-row tiles of probe rows per slice.
int fused_chunk_len(int max_tokens, int max_row_tiles);

}  // namespace tc
}  // namespace ckv
