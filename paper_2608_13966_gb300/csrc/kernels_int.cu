// Instantiations of the integer-code kernel for one candidate-chunk count
// (QUASAR_NCH = 1, 2 or 4 chunks of 8 candidates); compiled once per value.
#include "recon_int.cuh"

#ifndef QUASAR_NCH
#error "QUASAR_NCH must be defined"
#endif

#define QUASAR_CAT2(a, b) a##b
#define QUASAR_CAT(a, b) QUASAR_CAT2(a, b)

namespace quasar {

// Kernel entry for group size 8*epl, one tensor or a batch of up to
// kMaxBatch tensors per launch, or nullptr if not built.
const void* QUASAR_CAT(int_kernel_nch, QUASAR_NCH)(int epl, bool batch)
{
    switch (epl) {
    case 4: return batch ? reinterpret_cast<const void*>(&k_recon_int<4, QUASAR_NCH, kMaxBatch>)
                         : reinterpret_cast<const void*>(&k_recon_int<4, QUASAR_NCH, 1>);
    case 8: return batch ? reinterpret_cast<const void*>(&k_recon_int<8, QUASAR_NCH, kMaxBatch>)
                         : reinterpret_cast<const void*>(&k_recon_int<8, QUASAR_NCH, 1>);
    case 16: return batch ? reinterpret_cast<const void*>(&k_recon_int<16, QUASAR_NCH, kMaxBatch>)
                          : reinterpret_cast<const void*>(&k_recon_int<16, QUASAR_NCH, 1>);
    case 32: return batch ? reinterpret_cast<const void*>(&k_recon_int<32, QUASAR_NCH, kMaxBatch>)
                          : reinterpret_cast<const void*>(&k_recon_int<32, QUASAR_NCH, 1>);
    default: return nullptr;
    }
}

}  // namespace quasar
