// Delta-encoded host batches: each request's prompt is its base request's prompt followed
// by its own delta tokens (an agentic turn extends the session's previous turn; the
// samples of a prompt group repeat one prompt).  After the deltas have been copied to the
// device, this kernel rebuilds the full token array of the batch, so the routing kernels
// see exactly the batch the encoding describes.  No counterpart in the paper: an input
// encoding of the host path.
//
// One warp per request: lane 0 walks the chain r -> base(r) -> ... -> root (its depth is
// checked on the host), then the warp copies the deltas root first, each as coalesced
// 128-byte warp stores.  The host computed the full offsets, and the chain's deltas add up
// to exactly the request's full length.
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr int kExpandWarps = 8;
}  // namespace

__global__ void __launch_bounds__(32 * kExpandWarps) k_delta_expand(DeltaArgs a) {
  __shared__ int32_t s_chain[kExpandWarps][kDeltaMaxDepth];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int r = blockIdx.x * kExpandWarps + wid; r < a.n; r += gridDim.x * kExpandWarps) {
    int depth = 0;
    if (lane == 0) {
      int e = r;
      while (e >= 0 && depth < kDeltaMaxDepth) {
        s_chain[wid][depth++] = e;
        e = a.base[e];
      }
    }
    depth = __shfl_sync(0xffffffffu, depth, 0);
    __syncwarp();
    int32_t* out = a.tokens + a.tok_off[r];
    const int64_t len = a.tok_off[r + 1] - a.tok_off[r];
    int64_t pos = 0;
    for (int i = depth - 1; i >= 0; --i) {
      const int e = s_chain[wid][i];
      const int64_t d0 = a.doff[e];
      int64_t d = a.doff[e + 1] - d0;
      if (pos + d > len) d = len - pos;  // never for a well-formed encoding (host-checked)
      const int32_t* src = a.dtok + d0;
      for (int64_t j = lane; j < d; j += 32) out[pos + j] = src[j];
      pos += d;
    }
    __syncwarp();
  }
}

void launch_delta_expand(const DeltaArgs& a, int num_sms, cudaStream_t st) {
  if (a.n <= 0) return;
  const int blocks = (a.n + kExpandWarps - 1) / kExpandWarps;
  const int grid = blocks < num_sms * 8 ? blocks : num_sms * 8;
  k_delta_expand<<<grid, 32 * kExpandWarps, 0, st>>>(a);
}

}  // namespace misat
