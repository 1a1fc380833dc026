// The attention kernels of launches without the fused cache rewrite, in a
// translation unit of their own (see attention_kernels.cuh).

#include "attention_kernels.cuh"

namespace archer {

int launch_fwd_plain(int D, int kind, cudaLaunchConfig_t lc, const CUtensorMap* m, const AttnParams& prm) {
  if (D == 128) return launch_fwd<128, false>(kind, lc, m, prm);
  return launch_fwd<64, false>(kind, lc, m, prm);
}

}  // namespace archer
