// selftest.cu -- a diagnostic for the bounded waits every kernel of the
// library relies on. One warp waits, each time with a short limit, on
// things that never complete:
//   1. the globaltimer-bounded mbarrier wait of the tensor-core kernels;
//   2. the iteration-bounded mbarrier wait of the streaming kernels;
//   3. a flag spin as in the decoupled look-backs.
// Every wait must give up, the kernel records OCCAM_ERR_TIMEOUT in the status
// word and returns normally, so the CUDA context stays usable. Nothing here
// faults, traps or hangs: no asynchronous copy is in flight, and the only
// barrier is one the warp initialised itself.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

__global__ void __launch_bounds__(32) selftest_wait_kernel(uint64_t limit_ns, uint32_t max_iter, int32_t* out) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    tc::bar_init(&bar, 1);  // one arrival completes the phase; none ever comes
    tc::bar_fence_init();
  }
  __syncwarp();
  int gave_up = 0;
  if (!tc::bar_wait(&bar, 0, nullptr, limit_ns)) gave_up |= 1;
  if (!mbar_wait(&bar, 0, max_iter)) gave_up |= 2;
  const unsigned long long* flag = reinterpret_cast<const unsigned long long*>(out + 2);
  bool seen = false;
  for (uint32_t it = 0; it < max_iter && !seen; ++it) {
    seen = ld_acquire_u64(flag) != 0;
    if (!seen) __nanosleep(32);
  }
  if (!seen) gave_up |= 4;
  if (threadIdx.x == 0) {
    out[0] = gave_up;
    if (gave_up) set_status(out + 1, OCCAM_ERR_TIMEOUT);
  }
}

}  // namespace occam

extern "C" int occam_selftest_wait(uint64_t limit_ns, int32_t* scratch, occam_stream_t stream) {
  using namespace occam;
  if (!scratch || limit_ns == 0 || limit_ns > 1000000000ull) return OCCAM_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(scratch, 0, 16, st) != cudaSuccess) return OCCAM_ERR_CUDA;
  // about one try per 32 ns sleep: the iteration limit spans a similar time
  const uint32_t max_iter = (uint32_t)std::min<uint64_t>(limit_ns / 32, 1u << 24);
  launch_counter() = 0;
  selftest_wait_kernel<<<1, 32, 0, st>>>(limit_ns, max_iter < 16 ? 16 : max_iter, scratch);
  count_launch();
  return cudaGetLastError() == cudaSuccess ? OCCAM_OK : OCCAM_ERR_CUDA;
}
