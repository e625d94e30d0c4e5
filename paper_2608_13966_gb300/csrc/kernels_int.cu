// Instantiations of the integer-code kernel for one candidate-chunk count
// (QUASAR_NCH = 1, 2 or 4 chunks of 8 candidates) and one clamp-set size
// (QUASAR_SS = 4, 2 or 1 candidates; with a single chunk also 8, or 3 for
// the sets 3-3-2); compiled once per pair, in parallel.
#include "recon_int.cuh"

#if !defined(QUASAR_NCH) || !defined(QUASAR_SS)
#error "QUASAR_NCH and QUASAR_SS must be defined"
#endif

#define QUASAR_CAT4(a, b, c, d) a##b##c##d
#define QUASAR_NAME(n, s) QUASAR_CAT4(int_kernel_nch, n, _ss, s)

namespace quasar {

// Kernel entry for group size 4*epl: one tensor or a batch of up to
// kMaxBatch tensors per launch.  The AdamW-fused variant is built for batches
// with sets of 4 or 1 candidates, the option variants (var) for batches with
// sets of 1; nullptr where not built.
const void* QUASAR_NAME(QUASAR_NCH, QUASAR_SS)(int epl, bool batch, bool adam, bool var)
{
    constexpr int C = QUASAR_NCH;
    constexpr int S = QUASAR_SS;
    constexpr int B = kMaxBatch;
    if ((adam || var) && !batch) return nullptr;
    if (adam && (S == 2 || S == 3 || S == 8)) return nullptr;
    if (var && S != 1) return nullptr;
    switch (epl) {
#if QUASAR_SS == 1
#define QUASAR_VAR(E)                                                                         \
    if (var)                                                                                  \
        return adam ? reinterpret_cast<const void*>(&k_recon_int<E, C, B, true, true, S>)     \
                    : reinterpret_cast<const void*>(&k_recon_int<E, C, B, false, true, S>);
#else
#define QUASAR_VAR(E)
#endif
#if QUASAR_SS == 4 || QUASAR_SS == 1
#define QUASAR_ADAM(E) \
    if (adam) return reinterpret_cast<const void*>(&k_recon_int<E, C, B, true, false, S>);
#else
#define QUASAR_ADAM(E)
#endif
#define QUASAR_EPL(E)                                                                         \
    case E:                                                                                   \
        QUASAR_VAR(E)                                                                         \
        QUASAR_ADAM(E)                                                                        \
        if (!batch) return reinterpret_cast<const void*>(&k_recon_int<E, C, 1, false, false, S>); \
        return reinterpret_cast<const void*>(&k_recon_int<E, C, B, false, false, S>);
    QUASAR_EPL(8)
    QUASAR_EPL(16)
    QUASAR_EPL(32)
    QUASAR_EPL(64)
#undef QUASAR_EPL
#undef QUASAR_ADAM
#undef QUASAR_VAR
    default: return nullptr;
    }
}

}  // namespace quasar
