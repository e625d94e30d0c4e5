// Instantiations of the integer-code kernel for one candidate-chunk count
// (QUASAR_NCH = 1, 2 or 4 chunks of 8 candidates); compiled once per value.
#include "recon_int.cuh"

#ifndef QUASAR_NCH
#error "QUASAR_NCH must be defined"
#endif

#define QUASAR_CAT2(a, b) a##b
#define QUASAR_CAT(a, b) QUASAR_CAT2(a, b)

namespace quasar {

// Kernel entry for group size 8*epl: one tensor or a batch of up to
// kMaxBatch tensors per launch; the AdamW-fused variant and the option
// variants (var) are built for batches only.  nullptr if not built.
const void* QUASAR_CAT(int_kernel_nch, QUASAR_NCH)(int epl, bool batch, bool adam, bool var)
{
    constexpr int C = QUASAR_NCH;
    constexpr int B = kMaxBatch;
    if ((adam || var) && !batch) return nullptr;
    switch (epl) {
#define QUASAR_EPL(E)                                                                          \
    case E:                                                                                    \
        if (!batch) return reinterpret_cast<const void*>(&k_recon_int<E, C, 1, false, false>); \
        if (adam)                                                                              \
            return var ? reinterpret_cast<const void*>(&k_recon_int<E, C, B, true, true>)      \
                       : reinterpret_cast<const void*>(&k_recon_int<E, C, B, true, false>);    \
        return var ? reinterpret_cast<const void*>(&k_recon_int<E, C, B, false, true>)         \
                   : reinterpret_cast<const void*>(&k_recon_int<E, C, B, false, false>);
    QUASAR_EPL(4)
    QUASAR_EPL(8)
    QUASAR_EPL(16)
    QUASAR_EPL(32)
#undef QUASAR_EPL
    default: return nullptr;
    }
}

}  // namespace quasar
