// contract_tc.cu -- tcgen05 tile contraction (placeholder until the kernel lands).
#include "internal.cuh"

namespace ucl {

bool tc_supported(const TcPlan &, const ContractArgs &, std::string *why) {
    *why = "tcgen05 kernel not built";
    return false;
}

int tc_units(ucl_ctx *ctx, const TcPlan &, int64_t P) { return (int)(P < ctx->sm_count ? P : ctx->sm_count); }

ucl_status launch_contract_tc(ucl_ctx *ctx, const ContractArgs &, const TcPlan &, const ucl_rel *, const ucl_rel *) {
    return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 kernel not built");
}

}  // namespace ucl
