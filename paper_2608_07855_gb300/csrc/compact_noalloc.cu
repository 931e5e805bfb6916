// commitkv_compact_noalloc: the compression checkpoint of commitkv_compact
// (selection + gather) with its scratch memory in a fixed device array of
// this library instead of a caller-allocated workspace.
//
// Who needs it: code that cannot call cudaMalloc where it compacts.  A
// serving engine typically reserves nearly all device memory for its own KV
// pool at start-up, so a later cudaMalloc may fail or must go through the
// engine's allocator, which a plug-in may not reach; and cudaFree
// synchronises the whole device, which stalls every other stream of a
// latency-bound decode loop.  Such callers still own and pass every input
// and output; only the scratch (a 256-byte status header plus one class
// byte per resident token) lives here.
//
// The array below exists once on every GPU that loads this library and stays
// there until the process exits.  Every call on a GPU uses the same array:
// calls that can overlap on that GPU (two streams, two host threads) race on
// it and must be serialised by the caller.
#include <atomic>
#include <string.h>

#include "ckv_internal.cuh"

using namespace ckv;

namespace {

constexpr size_t kScratchBytes = COMMITKV_NOALLOC_SCRATCH_BYTES;
constexpr size_t kAlign = 256;
constexpr int kMaxDevices = 64;

static_assert(kScratchBytes % kAlign == 0, "scratch size is a multiple of 256 bytes");

// Scratch of every commitkv_compact_noalloc call on this device: a WsHeader
// (status word, cleared at the start of each call), then one class byte per
// resident token of each trajectory (every byte is written by the selection
// kernel before it is read, so these need no clearing).
static __device__ __align__(256) unsigned char g_compact_scratch[kScratchBytes];

// Device address of g_compact_scratch per device, filled on the first call
// made with that device current.  In host code the array's name is only a
// host-side stand-in, so the address must come from cudaGetSymbolAddress.
std::atomic<void *> g_scratch_addr[kMaxDevices];

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

commitkv_status scratch_for_current_device(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return COMMITKV_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) return COMMITKV_ERR_UNSUPPORTED;
  void *p = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (!p) {
    // Two threads may both get here; they store the same address.
    if (cudaGetSymbolAddress(&p, g_compact_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return COMMITKV_ERR_CUDA;
    }
    g_scratch_addr[dev].store(p, std::memory_order_release);
  }
  *out = p;
  return COMMITKV_OK;
}

}  // namespace

extern "C" commitkv_status commitkv_compact_noalloc(
    const commitkv_shape *shape, int32_t n_traj, const commitkv_traj *cache,
    const uint8_t *const *retired, const int32_t *const *pending, const int32_t *n_pending,
    const float *const *pending_priority, const float *const *fill_score, int32_t budget_B,
    int32_t pending_tokens_BN, int32_t pending_cap_pages, int32_t *const *idx_out,
    int32_t *n_idx_out, void *const *k_out, void *const *v_out, int32_t *const *pos_out,
    int32_t *status_out, cudaStream_t stream) {
  // the host-side checks of commitkv_compact, shared with it
  commitkv_status st = check_compact_args(shape, n_traj, cache, retired, pending, n_pending,
                                          pending_priority, fill_score, budget_B, pending_tokens_BN,
                                          pending_cap_pages, idx_out, n_idx_out);
  if (st) return st;
  // Sizes beyond the fixed array are refused before anything is launched.
  size_t need = kAlign;
  for (int t = 0; t < n_traj; ++t) need += align_up((size_t)cache[t].S);
  if (need > kScratchBytes) return COMMITKV_ERR_WORKSPACE;

  void *scratch = nullptr;
  if ((st = scratch_for_current_device(&scratch))) return st;
  WsHeader *hdr = static_cast<WsHeader *>(scratch);

  static thread_local CompactLaunch L;
  memset(&L, 0, sizeof L);
  L.n_traj = n_traj;
  L.M = shape->layers;
  L.H = shape->kv_heads;
  L.d = shape->head_dim;
  L.elem_bytes = shape->dtype == COMMITKV_BF16 ? 2 : 4;
  char *base = static_cast<char *>(scratch) + kAlign;
  for (int t = 0; t < n_traj; ++t) {
    const commitkv_traj &x = cache[t];
    TrajDev &d = L.t[t];
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
    L.retired[t] = retired[t];
    L.pending[t] = n_pending[t] ? pending[t] : nullptr;
    L.n_pending[t] = n_pending[t];
    L.prio[t] = n_pending[t] ? pending_priority[t] : nullptr;
    L.fill[t] = fill_score[t];
    L.cls[t] = reinterpret_cast<uint8_t *>(base);
    base += align_up((size_t)x.S);
    L.idx[t] = idx_out[t];
    L.k_out[t] = k_out ? k_out[t] : nullptr;
    L.v_out[t] = v_out ? v_out[t] : nullptr;
    L.pos_out[t] = pos_out ? pos_out[t] : nullptr;
  }
  L.n_idx = n_idx_out;
  L.B = budget_B;
  L.B_N = pending_tokens_BN;
  L.cap = pending_cap_pages;

  // The status word keeps the previous call's value: clear the header.
  cudaError_t e = cudaMemsetAsync(hdr, 0, sizeof(WsHeader), stream);
  if (e == cudaSuccess) e = launch_compact(L, hdr, stream);
  if (e == cudaSuccess && status_out)
    e = cudaMemcpyAsync(status_out, &hdr->status, sizeof(int32_t), cudaMemcpyDeviceToDevice, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return COMMITKV_ERR_CUDA;
  }
  return COMMITKV_OK;
}
