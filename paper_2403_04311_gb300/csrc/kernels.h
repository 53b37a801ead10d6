// Host-side launch interfaces shared between the library's translation units.
#pragma once

#include <utility>

#include "common.cuh"

namespace alto {

// Launch with programmatic stream serialization: the kernel may be scheduled
// while its predecessor finishes and waits for it in pdl_enter().
template <typename... KArgs, typename... Args>
inline void launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

struct SortBuffers {
  u32* keys[2];
  u32* vals[2];
  u32* hist;      // [4][256], zero between sorts
  u32* bin_base;  // [4][256]
  u64* lookback;  // [lb_tiles][256]
  u64 lb_tiles;
};

// Stable sort of keys[0] (values: identity when vals_identity, else vals[0])
// by the low `bits` bits; the element count is read from n_dev on the device
// and clamped to n_cap.  Returns the index (0/1) of the buffers holding the
// result.  Uses launch sites site_base .. site_base + passes - 1.
// A capacity of at most 8,192 pairs is sorted by one CTA in shared memory
// (sort_prepare must have run on the device), a larger one by onesweep passes.
int sort_pairs(const u32* n_dev, u32 n_cap, int bits, bool vals_identity, SortBuffers& b,
               Ctl* ctl, int site_base, u64 spin_limit, int num_sms, cudaStream_t s,
               int* launches);

// Once per device before the first sort: the one-CTA sort's shared memory.
cudaError_t sort_prepare();

}  // namespace alto
