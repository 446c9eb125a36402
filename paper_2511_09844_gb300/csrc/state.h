// Launchers of the device-side bookkeeping kernels (row plans, commit/rollback, prefill init).
#pragma once

#include <cuda_runtime.h>

namespace sd2 {

enum PlanMode { PLAN_DRAFT_FIRST = 0, PLAN_DRAFT_NEXT = 1, PLAN_VERIFY = 2 };

// state: [4][maxB] int32 rows (n committed, drafter cached length, last j, stopped).
cudaError_t plan_rows(int mode, int i, int B, int k, int max_ctx, const int* state, int maxB, const int* committed,
                      const int* xhat, int* tok, int* pos, int* seq, int* valid, cudaStream_t st);
cudaError_t commit(int B, int k, int max_ctx, int* state, int maxB, int* committed, const int* tokens, const int* n_out,
                   int* iter, cudaStream_t st);
cudaError_t prefill_init(int B, int max_ctx, const int* prompts, const int* cu, const int* first, int* state, int maxB,
                         int* committed, int* first_out, cudaStream_t st);
// One bounded device wait that nothing satisfies: gives up after `cycles` clock cycles and
// latches ERR_TIMEOUT in *err (failure-detection test of the bounded waits).
cudaError_t expire_wait(unsigned* err, long long cycles, cudaStream_t st);

}  // namespace sd2
