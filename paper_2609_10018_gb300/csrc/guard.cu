// Guard zones around arena sub-buffers: fill at create time, check on demand
// (see guard.h).
#include "guard.h"

namespace elasto {

namespace {

// One block per zone, threads striding over its bytes.
__global__ void guard_fill_kernel(char* base, const unsigned long long* off, const unsigned long long* len) {
  const int z = blockIdx.x;
  unsigned char* p = reinterpret_cast<unsigned char*>(base + off[z]);
  for (unsigned long long i = threadIdx.x; i < len[z]; i += blockDim.x) p[i] = kGuardByte;
}

__global__ void guard_check_kernel(const char* base, const unsigned long long* off, const unsigned long long* len,
                                   unsigned int* bad) {
  const int z = blockIdx.x;
  const unsigned char* p = reinterpret_cast<const unsigned char*>(base + off[z]);
  unsigned int n = 0;
  for (unsigned long long i = threadIdx.x; i < len[z]; i += blockDim.x) n += p[i] != kGuardByte ? 1u : 0u;
  if (n) atomicAdd(&bad[z], n);
}

}  // namespace

cudaError_t guard_fill_launch(char* base, const unsigned long long* off, const unsigned long long* len, int nz,
                              cudaStream_t s) {
  if (nz <= 0) return cudaSuccess;
  guard_fill_kernel<<<nz, 256, 0, s>>>(base, off, len);
  return cudaGetLastError();
}

cudaError_t guard_check_launch(const char* base, const unsigned long long* off, const unsigned long long* len, int nz,
                               unsigned int* bad, cudaStream_t s) {
  if (nz <= 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(bad, 0, sizeof(unsigned int) * nz, s);
  if (e != cudaSuccess) return e;
  guard_check_kernel<<<nz, 256, 0, s>>>(base, off, len, bad);
  return cudaGetLastError();
}

elasto_status GuardedArena::upload(char* base) {
  const int nz = static_cast<int>(zones.size());
  if (nz == 0) return ELASTO_OK;
  std::vector<unsigned long long> ho(nz), hl(nz);
  for (int z = 0; z < nz; ++z) {
    ho[z] = zones[z].off;
    hl[z] = zones[z].bytes;
  }
  const size_t tb = sizeof(unsigned long long) * nz;
  char* buf = nullptr;
  cudaError_t e = cudaMalloc(&buf, 2 * tb + sizeof(unsigned int) * nz);
  if (e != cudaSuccess) {
    cudaGetLastError();
    set_error("guard zones: cudaMalloc of the zone table failed");
    return ELASTO_ERR_OOM;
  }
  d_off = reinterpret_cast<unsigned long long*>(buf);
  d_len = reinterpret_cast<unsigned long long*>(buf + tb);
  d_bad = reinterpret_cast<unsigned int*>(buf + 2 * tb);
  ELASTO_CUDA_TRY(cudaMemcpy(d_off, ho.data(), tb, cudaMemcpyHostToDevice));
  ELASTO_CUDA_TRY(cudaMemcpy(d_len, hl.data(), tb, cudaMemcpyHostToDevice));
  ELASTO_CUDA_TRY(guard_fill_launch(base, d_off, d_len, nz, 0));
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());
  return ELASTO_OK;
}

int GuardedArena::check(char* base, cudaStream_t s, std::string* first_bad) const {
  const int nz = static_cast<int>(zones.size());
  if (nz == 0 || !d_off) return 0;
  if (guard_check_launch(base, d_off, d_len, nz, d_bad, s) != cudaSuccess) return -1;
  std::vector<unsigned int> hb(nz);
  if (cudaMemcpyAsync(hb.data(), d_bad, sizeof(unsigned int) * nz, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return -1;
  int bad = 0;
  for (int z = 0; z < nz; ++z)
    if (hb[z]) {
      if (bad == 0 && first_bad)
        *first_bad = zones[z].name + " (" + std::to_string(hb[z]) + " of " + std::to_string(zones[z].bytes) +
                     " guard bytes after it changed)";
      ++bad;
    }
  return bad;
}

void GuardedArena::release() {
  if (d_off) cudaFree(d_off);
  d_off = nullptr;
  d_len = nullptr;
  d_bad = nullptr;
}

}  // namespace elasto
