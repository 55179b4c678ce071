// Device side of the seeded synthetic input generators (see synth/__init__.py).
//
// Integer-only expansions of the counter-based generator, producing the same bytes as
// the numpy implementation: a value is mix(row_key + (i + 1) * GOLDEN), where the host
// precomputes row_key = mix(stream_key(seed, purpose) + (a + 1) * GOLDEN) for every row a,
// and mix is SplitMix64's output function.  Holds no part of the scoring method.
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t nonzero(uint64_t x) { return x ? x : kGolden; }

// chain of request r: blocks [0, shared[r]) from root_key[r], the rest from tail_key[r]
__global__ void chains_kernel(uint64_t* out, const uint64_t* off, const uint64_t* root_key,
                              const uint64_t* tail_key, const uint32_t* shared, uint64_t R) {
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t lane = threadIdx.x & 31;
  for (uint64_t r = warp; r < R; r += n_warps) {
    const uint64_t b = off[r], n = off[r + 1] - b;
    const uint64_t sh = shared[r], rk = root_key[r], tk = tail_key[r];
    for (uint64_t i = lane; i < n; i += 32)
      out[b + i] = nonzero(mix((i < sh ? rk : tk) + (i + 1) * kGolden));
  }
}

// keys of table t: segment s in [0, n_seg) covers [cum[t][s], cum[t][s+1]) with row key
// seg_key[t][s]; element j of a segment is the (j - cum[t][s])-th value of that row.
__global__ void keys_kernel(uint64_t* out, uint64_t n_tables, uint32_t n_seg, uint64_t n_keys,
                            const uint64_t* seg_key, const uint64_t* cum) {
  for (uint64_t t = blockIdx.x; t < n_tables; t += gridDim.x) {
    const uint64_t* c = cum + t * (n_seg + 1);
    const uint64_t* k = seg_key + t * n_seg;
    for (uint64_t j = threadIdx.x; j < n_keys; j += blockDim.x) {
      uint32_t lo = 0, hi = n_seg;  // c[lo] <= j < c[hi]
      while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (c[mid] <= j) lo = mid; else hi = mid;
      }
      out[t * n_keys + j] = nonzero(mix(k[lo] + (j - c[lo] + 1) * kGolden));
    }
  }
}

// uniform utilisation in [0, 0.9): m = floor(top24 * 9 / 10), u = m * 2^-24 (exact)
__global__ void util_kernel(float* out, uint64_t n_rows, uint32_t n_cols, const uint64_t* row_key) {
  const uint64_t total = n_rows * n_cols;
  for (uint64_t idx = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t s = idx / n_cols, e = idx - s * n_cols;
    const uint64_t x = mix(row_key[s] + (e + 1) * kGolden);
    const uint64_t m = ((x >> 40) * 9) / 10;
    out[idx] = (float)m * 5.9604644775390625e-08f;
  }
}

unsigned grid_for(uint64_t work, uint64_t per_block) {
  const uint64_t b = (work + per_block - 1) / per_block;
  return (unsigned)(b < (1u << 20) ? (b ? b : 1) : (1u << 20));
}

}  // namespace

extern "C" int synth_chains(uint64_t* out, const uint64_t* off, const uint64_t* root_key,
                            const uint64_t* tail_key, const uint32_t* shared, uint64_t R,
                            void* stream) {
  if (R == 0) return 0;
  chains_kernel<<<grid_for(R, 8), 256, 0, (cudaStream_t)stream>>>(out, off, root_key, tail_key,
                                                                   shared, R);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

extern "C" int synth_keys(uint64_t* out, uint64_t n_tables, uint32_t n_seg, uint64_t n_keys,
                          const uint64_t* seg_key, const uint64_t* cum, void* stream) {
  if (n_tables == 0 || n_keys == 0) return 0;
  const unsigned grid = (unsigned)(n_tables < (1u << 20) ? n_tables : (1u << 20));
  keys_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(out, n_tables, n_seg, n_keys, seg_key, cum);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}

extern "C" int synth_util_uniform09(float* out, uint64_t n_rows, uint32_t n_cols,
                                    const uint64_t* row_key, void* stream) {
  if (n_rows == 0 || n_cols == 0) return 0;
  util_kernel<<<grid_for(n_rows * n_cols, 256), 256, 0, (cudaStream_t)stream>>>(out, n_rows, n_cols,
                                                                                 row_key);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : 3;
}
