// tqfx4_selftest_wait_timeout: exercises the failure detection of the
// streaming engine (tq_stream.cuh) without a fault. One warp runs the
// engine's consume loop on a ring whose copies were never issued, so the
// wait on its first slot cannot complete; with a budget of 10^6 cycles
// (about half a millisecond) instead of the production two seconds, the
// wait gives up, the warp records TQFX4_ETIMEOUT in the status word and the
// kernel returns. Nothing is in flight when it gives up (no copy was issued),
// so the context stays usable and the next call runs normally.
#include "tq_launch.h"
#include "tq_stream.cuh"

namespace tq {

namespace {

constexpr long long kSelftestBudget = 1000000LL;

__global__ void __launch_bounds__(32) selftest_timeout_kernel(int *status) {
    __shared__ __align__(128) uint8_t smem[1280];  // one 1056-byte slot, its sums and its barrier
    const int nb = 2, rpu = 1;  // a job of one unit: one row group of two blocks
    const WarpRing ring = carve_ring(smem, 1, stream_slot_bytes(rpu, nb), rpu, nb);
    WarpRing r = ring;
    r.budget = kSelftestBudget;
    ring_init(r);
    fence_barrier_init();
    __syncwarp();
    __shared__ uint8_t qs[2 * QS_STRIDE];
    __shared__ float das[2];
    __shared__ int bss[2];
    MatJob job;
    job.mat = nullptr;  // never dereferenced: the unit's copy is not issued and the wait gives up first
    job.rg_begin = 0;
    job.rg_end = 1;
    job.y = nullptr;
    job.s_out = nullptr;
    job.qs = qs;
    job.das = das;
    job.bss = bss;
    job.nb = nb;
    warp_stream_run(r, job, rpu, 0, 1, status, K_SELFTEST);
}

}  // namespace

cudaError_t launch_selftest_timeout(int *status, cudaStream_t st) {
    selftest_timeout_kernel<<<1, 32, 0, st>>>(status);
    return cudaGetLastError();
}

}  // namespace tq
