// Global prefix index maintenance outside the commit path: rebuild from the instance
// tables, and the clear that precedes an instance reset (Sec. 4.4: a cache reset removes
// the instance from every hash it held).
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace misat {

// grid (chunks, W): chunk x of instance w's buckets.
__global__ void __launch_bounds__(256) k_gix_build(const InstDesc* desc, GIndex g, int32_t* err) {
  if (block_error(err)) return;
  const int w = blockIdx.y;
  const InstDesc d = desc[w];
  const uint32_t NB = 1u << d.log2nb;
  long long claimed = 0;
  for (uint32_t b = blockIdx.x * blockDim.x + threadIdx.x; b < NB; b += gridDim.x * blockDim.x) {
    unsigned long long k[4];
    ld_bucket_keys(d.tab + b, k);
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      if (k[s] == kEmpty) continue;
      const int r = gix_set(g, k[s], w);
      if (r < 0)
        set_error(err, MISAT_ERR_TABLE_FULL);
      else
        claimed += r;
    }
  }
  const long long tot = block_sum(claimed);
  if (threadIdx.x == 0 && tot) atomicAdd(g.used, (unsigned long long)tot);
}

void launch_gix_build(const InstDesc* desc, int32_t W, uint32_t max_log2nb, const GIndex& g, int32_t* err,
                      cudaStream_t st) {
  if (W <= 0) return;
  const uint64_t nb = 1ull << max_log2nb;
  const int chunks = (int)std::min<uint64_t>(256, std::max<uint64_t>(1, nb / 1024));
  k_gix_build<<<dim3(chunks, W), 256, 0, st>>>(desc, g, err);
}

__global__ void __launch_bounds__(256) k_gix_clear_table(InstDesc d, int32_t w, GIndex g, int32_t* err) {
  const uint32_t NB = 1u << d.log2nb;
  for (uint32_t b = blockIdx.x * blockDim.x + threadIdx.x; b < NB; b += gridDim.x * blockDim.x) {
    unsigned long long k[4];
    ld_bucket_keys(d.tab + b, k);
#pragma unroll
    for (int s = 0; s < 4; ++s)
      if (k[s] != kEmpty && gix_clear(g, k[s], w) < 0) set_error(err, MISAT_ERR_INTERNAL);
  }
}

void launch_gix_clear_table(const InstDesc& d, int32_t w, const GIndex& g, int32_t* err, cudaStream_t st) {
  const uint32_t NB = 1u << d.log2nb;
  const uint32_t blocks = (NB + 255) / 256;
  k_gix_clear_table<<<blocks < 4096 ? blocks : 4096, 256, 0, st>>>(d, w, g, err);
}

}  // namespace misat
