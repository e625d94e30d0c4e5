// Instantiations of the symmetric integer-code kernel (batches of up to
// kMaxBatch tensors; one tensor is a batch of one), group size 8*epl.
#include "recon_sym.cuh"

namespace quasar {

const void* sym_kernel(int epl)
{
    switch (epl) {
    case 4: return reinterpret_cast<const void*>(&k_recon_sym<4, kMaxBatch>);
    case 8: return reinterpret_cast<const void*>(&k_recon_sym<8, kMaxBatch>);
    case 16: return reinterpret_cast<const void*>(&k_recon_sym<16, kMaxBatch>);
    case 32: return reinterpret_cast<const void*>(&k_recon_sym<32, kMaxBatch>);
    default: return nullptr;
    }
}

}  // namespace quasar
