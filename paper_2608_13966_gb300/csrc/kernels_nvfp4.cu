// Instantiations of the NVFP4 kernel (1, 2 or 4 chunks of 8 candidates) and
// of the tensor-absmax kernels.
#include "recon_adamw.cuh"
#include "recon_nvfp4.cuh"

namespace quasar {

const void* nvfp4_kernel(int nch, bool batch)
{
    switch (nch) {
    case 1: return batch ? reinterpret_cast<const void*>(&k_recon_nvfp4<1, kMaxBatch>)
                         : reinterpret_cast<const void*>(&k_recon_nvfp4<1, 1>);
    case 2: return batch ? reinterpret_cast<const void*>(&k_recon_nvfp4<2, kMaxBatch>)
                         : reinterpret_cast<const void*>(&k_recon_nvfp4<2, 1>);
    case 4: return batch ? reinterpret_cast<const void*>(&k_recon_nvfp4<4, kMaxBatch>)
                         : reinterpret_cast<const void*>(&k_recon_nvfp4<4, 1>);
    default: return nullptr;
    }
}

const void* amax_kernel(bool batch)
{
    return batch ? reinterpret_cast<const void*>(&k_amax<kMaxBatch>)
                 : reinterpret_cast<const void*>(&k_amax<1>);
}

const void* adamw_amax_kernel() { return reinterpret_cast<const void*>(&k_adamw_amax<kMaxBatch>); }

const void* amax_init_kernel(bool batch)
{
    return batch ? reinterpret_cast<const void*>(&k_amax_init<kMaxBatch>)
                 : reinterpret_cast<const void*>(&k_amax_init<1>);
}

const void* amax_to_scale_kernel(bool batch)
{
    return batch ? reinterpret_cast<const void*>(&k_amax_to_scale<kMaxBatch>)
                 : reinterpret_cast<const void*>(&k_amax_to_scale<1>);
}

}  // namespace quasar
