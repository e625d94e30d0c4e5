// Instantiations of the NVFP4 kernel (1, 2 or 4 chunks of 8 candidates) and
// of the tensor-absmax kernels.
#include "recon_nvfp4.cuh"

namespace quasar {

const void* nvfp4_kernel(int nch)
{
    switch (nch) {
    case 1: return reinterpret_cast<const void*>(&k_recon_nvfp4<1>);
    case 2: return reinterpret_cast<const void*>(&k_recon_nvfp4<2>);
    case 4: return reinterpret_cast<const void*>(&k_recon_nvfp4<4>);
    default: return nullptr;
    }
}

const void* amax_kernel() { return reinterpret_cast<const void*>(&k_amax); }
const void* amax_to_scale_kernel() { return reinterpret_cast<const void*>(&k_amax_to_scale); }

}  // namespace quasar
