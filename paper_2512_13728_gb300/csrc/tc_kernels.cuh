// Launch wrappers of the tcgen05 kernels (tc_bq.cu, tc.cu).
#pragma once

#include "common.cuh"
#include "tc.cuh"

namespace cd {
namespace tc {

uint32_t form_bq_smem(int nstages, uint32_t stage_bytes);
uint32_t btp_smem(int nstages, uint32_t stage_bytes);
cudaError_t setup_bq_kernels(uint32_t f_smem, uint32_t r_smem, bool x3);
void launch_form_bq(const Shared &sh, const TcPlan &tp, cudaStream_t s);
uint32_t fused_bq_smem(uint32_t bq_boxes);
cudaError_t setup_fused_bq_kernel(uint32_t smem);
void launch_fused_bq(const Shared &sh, const TcPlan &tp, bool gated, cudaStream_t s);
void launch_btp(const Shared &sh, const TcPlan &tp, cudaStream_t s);
// data-parallel phases: P_raw^T from the averaged P_raw; R's bf16 copies and column partials
// from the averaged R
void launch_transpose_praw(const Shared &sh, const TcPlan &tp, cudaStream_t s);
void launch_r_refresh(const Shared &sh, const TcPlan &tp, cudaStream_t s);
void launch_qn_refresh(const Shared &sh, const TcPlan &tp, cudaStream_t s);
void launch_colnorm_reduce(const Shared &sh, const int4 *ctiles, int32_t n_ctiles, float eps_col, cudaStream_t s);
void launch_colnorm_scale(const Shared &sh, const TcPlan &tp, cudaStream_t s);
uint32_t orth_smem(int nstages, uint32_t stage_bytes);
cudaError_t setup_orth_kernels(uint32_t smem, bool x3);
void launch_orth(const Shared &sh, const TcPlan &tp, bool gram, int pass, cudaStream_t s);
cudaError_t setup_update_kernel(bool x3);
void launch_update(const Shared &sh, const TcPlan &tp, float mu, float eta, float keep, cudaStream_t s);

}  // namespace tc
}  // namespace cd
