// The attention kernels of launches with the fused cache rewrite, in a
// translation unit of their own (see attention_kernels.cuh).

#include "attention_kernels.cuh"

namespace archer {

int launch_fwd_rewrite(int D, int kind, cudaLaunchConfig_t lc, const CUtensorMap* m, const AttnParams& prm) {
  if (D == 128) return launch_fwd<128, true>(kind, lc, m, prm);
  return launch_fwd<64, true>(kind, lc, m, prm);
}

}  // namespace archer
