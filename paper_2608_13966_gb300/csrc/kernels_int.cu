// Instantiations of the integer-code kernel for one candidate-chunk count
// (QUASAR_NCH = 1, 2 or 4 chunks of 8 candidates); compiled once per value,
// and once more with QUASAR_HC for the hoisted-clamp variant (one chunk).
#include "recon_int.cuh"

#ifndef QUASAR_NCH
#error "QUASAR_NCH must be defined"
#endif

#define QUASAR_CAT2(a, b) a##b
#define QUASAR_CAT(a, b) QUASAR_CAT2(a, b)

namespace quasar {

#ifdef QUASAR_HC
// Kernel entry of the hoisted-clamp variant (batches of up to kMaxBatch
// tensors, one chunk of 8 candidates, no option variants); nullptr if not
// built.
const void* int_kernel_hc(int epl, bool adam)
{
    constexpr int B = kMaxBatch;
    switch (epl) {
#define QUASAR_EPL(E)                                                                       \
    case E:                                                                                 \
        return adam ? reinterpret_cast<const void*>(&k_recon_int<E, 1, B, true, false, true>) \
                    : reinterpret_cast<const void*>(&k_recon_int<E, 1, B, false, false, true>);
    QUASAR_EPL(4)
    QUASAR_EPL(8)
    QUASAR_EPL(16)
    QUASAR_EPL(32)
#undef QUASAR_EPL
    default: return nullptr;
    }
}
#else
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
#endif

}  // namespace quasar
