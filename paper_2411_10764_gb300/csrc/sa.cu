// Explorer proposal step on the device: one simulated-annealing move for
// each of m chains through the knob space.
//
// ML^2Tuner Sec. 2 ("Configuration Explorer"): the explorer searches the
// space of configurations and keeps those the models rank highest; the
// search algorithm itself is left open (TVM's explorer anneals).  A move
// mutates one knob of a chain's current configuration (knob and new option
// index taken from random words the caller draws), the proposal is decoded
// and screened by V and P like any candidate (decode_column + the walk
// kernels), and the Metropolis rule keeps it iff it is valid and
//   fl(score - parent_score) >= fl(temperature * ln u)
// with ln u passed in, so the decision is a plain float comparison.
#include "mlt_internal.cuh"

namespace mlt {
namespace {

__global__ void k_sa_propose(const __grid_constant__ DecodeParams d, long long space, const int64_t* parent,
                             const uint32_t* knob_draw, const uint32_t* digit_draw, long long m, long long* prop,
                             unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= m) return;
  const long long p = parent[i];
  if (p < 0 || p >= space) {
    if (p >= space) atomicOr(err, kErrBadIndex);
    prop[i] = 0;  // inactive chain: a harmless stand-in, ignored at acceptance
    return;
  }
  const int kj = static_cast<int>(knob_draw[i] % static_cast<uint32_t>(d.n_knobs));
  long long rem = p, place = 1, q = 0;
  for (int j = 0; j < d.n_knobs; ++j) {
    const long long r = d.radix[j];
    const long long next = rem / r;
    long long digit = rem - next * r;
    rem = next;
    if (j == kj) digit = static_cast<long long>(digit_draw[i] % static_cast<uint32_t>(r));
    q += digit * place;
    place *= r;
  }
  prop[i] = q;
}

__global__ void k_sa_accept(long long space, const int64_t* parent, const float* parent_score,
                            const long long* prop, const float* perf, const float* log_u, long long m,
                            float temperature, int64_t* out_next, float* out_next_score, int32_t* out_accepted) {
  pdl_wait();
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= m) return;
  const long long p = parent[i];
  const float ps = parent_score[i];
  bool accept = false;
  float s = -INFINITY;
  if (p >= 0 && p < space) {
    s = perf[i];
    if (s != -INFINITY) accept = __fsub_rn(s, ps) >= __fmul_rn(temperature, log_u[i]);
  }
  out_next[i] = accept ? prop[i] : p;
  out_next_score[i] = accept ? s : ps;
  out_accepted[i] = accept ? 1 : 0;
}

}  // namespace

cudaError_t launch_sa_propose(const DecodeParams& dec, long long space, const int64_t* parent,
                              const uint32_t* knob_draw, const uint32_t* digit_draw, long long m, long long* prop,
                              unsigned* err, cudaStream_t st) {
  if (m <= 0) return cudaSuccess;
  const unsigned grid = static_cast<unsigned>((m + 255) / 256);
  return launch_pdl(k_sa_propose, dim3(grid), dim3(256), 0, st, dec, space, parent, knob_draw, digit_draw, m, prop,
                    err);
}

cudaError_t launch_sa_accept(long long space, const int64_t* parent, const float* parent_score, const long long* prop,
                             const float* perf, const float* log_u, long long m, float temperature, int64_t* out_next,
                             float* out_next_score, int32_t* out_accepted, cudaStream_t st) {
  if (m <= 0) return cudaSuccess;
  const unsigned grid = static_cast<unsigned>((m + 255) / 256);
  return launch_pdl(k_sa_accept, dim3(grid), dim3(256), 0, st, space, parent, parent_score, prop, perf, log_u, m,
                    temperature, out_next, out_next_score, out_accepted);
}

}  // namespace mlt
