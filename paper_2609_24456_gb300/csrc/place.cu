// place.cu -- bandwidth-aware placement (Sec. 5): the transfer-latency model
// of Sec. 5.1, the feasible minimum of Eq. 1 by the linear scan of Alg. 1,
// and the placement map of Appendix D.  Host code only; the formulas are
// stated in edp.h.
#include <chrono>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <limits>

#include "edp_internal.cuh"

namespace {

bool pos(double v) { return std::isfinite(v) && v > 0.0; }

bool valid(const edp_place_option &o) {
  if (o.tiers != 1 && o.tiers != 2) return false;
  if (!pos(o.bw_in) || !pos(o.bw_out) || !std::isfinite(o.mem) || o.mem < 0.0) return false;
  if (o.tiers == 2 && (!pos(o.bw_out2) || !std::isfinite(o.mem2) || o.mem2 < 0.0))
    return false;
  return true;
}

// T(p, x), or +infinity when the buffer C_buf x does not fit
double transfer(const edp_place_option &o, double c_buf, double x) {
  const double need = c_buf * x;
  const double cap = o.tiers == 2 ? o.mem + o.mem2 : o.mem;
  if (need > cap) return std::numeric_limits<double>::infinity();
  double out = x / o.bw_out;
  if (o.tiers == 2) {
    const double h = o.mem >= need ? 1.0 : o.mem / need;  // share read from tier 1
    out = x * (h / o.bw_out + (1.0 - h) / o.bw_out2);
  }
  return x / o.bw_in + out;
}

// Alg. 1: the first feasible option with the smallest T; n if none
uint32_t scan(const edp_place_option *opts, uint32_t n, double c_buf, double x,
              double *t_all) {
  uint32_t best = n;
  double t_min = std::numeric_limits<double>::infinity();
  for (uint32_t i = 0; i < n; ++i) {
    const double t = transfer(opts[i], c_buf, x);
    if (t_all) t_all[i] = t;
    if (std::isfinite(t) && t < t_min) {
      t_min = t;
      best = i;
    }
  }
  return best;
}

bool valid_all(const edp_place_option *opts, uint32_t n, double c_buf) {
  if (!opts || n == 0 || !pos(c_buf)) return false;
  for (uint32_t i = 0; i < n; ++i)
    if (!valid(opts[i])) return false;
  return true;
}

}  // namespace

namespace {

// best of three: bytes / seconds of one timed call of f (GPU work timed with
// events on the legacy stream, synchronised)
template <typename F>
double best_gpu(uint64_t bytes, F f, cudaError_t *err) {
  cudaEvent_t a, b;
  cudaEventCreate(&a);
  cudaEventCreate(&b);
  double best = 0.0;
  f();  // warm
  for (int r = 0; r < 3 && *err == cudaSuccess; ++r) {
    cudaEventRecord(a);
    f();
    cudaEventRecord(b);
    *err = cudaEventSynchronize(b);
    float ms = 0.f;
    if (*err == cudaSuccess) *err = cudaEventElapsedTime(&ms, a, b);
    if (*err == cudaSuccess && ms > 0.f) {
      const double v = (double)bytes / (ms * 1e-3);
      if (v > best) best = v;
    }
  }
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  return best;
}

}  // namespace

extern "C" {

edp_status edp_place_choose(const edp_place_option *opts, uint32_t n, double c_buf,
                            double x, uint32_t *best, double *t_all) {
  if (!best || !valid_all(opts, n, c_buf) || !pos(x)) return EDP_ERR_INVALID;
  *best = scan(opts, n, c_buf, x, t_all);
  return *best < n ? EDP_OK : EDP_ERR_EMPTY;
}

edp_status edp_place_map(const edp_place_option *opts, uint32_t n, double c_buf,
                         const double *x, uint32_t nx, uint32_t *choice) {
  if (!x || !choice || !valid_all(opts, n, c_buf)) return EDP_ERR_INVALID;
  for (uint32_t i = 0; i < nx; ++i)
    if (!pos(x[i])) return EDP_ERR_INVALID;
  for (uint32_t i = 0; i < nx; ++i) choice[i] = scan(opts, n, c_buf, x[i], nullptr);
  return EDP_OK;
}

edp_status edp_place_profile(int device, uint64_t bytes, edp_place_bw *out) {
  if (!out || bytes < (1u << 20) || bytes % 16) return EDP_ERR_INVALID;
  if (cudaSetDevice(device) != cudaSuccess) {
    cudaGetLastError();
    return EDP_ERR_INVALID;
  }
  edp_place_bw r{};
  size_t free_b = 0, total_b = 0;
  cudaMemGetInfo(&free_b, &total_b);
  r.hbm_free = (double)free_b;
  uint8_t *d = nullptr, *pin = nullptr, *page = nullptr;
  uint64_t *fold = nullptr;
  edp_status st = EDP_OK;
  if (cudaMalloc(&d, 2 * bytes) != cudaSuccess || cudaMalloc(&fold, 16) != cudaSuccess ||
      cudaHostAlloc(&pin, bytes, cudaHostAllocMapped) != cudaSuccess) {
    cudaGetLastError();
    st = EDP_ERR_OOM;
  }
  if (st == EDP_OK && !(page = (uint8_t *)std::malloc(bytes))) st = EDP_ERR_OOM;
  cudaError_t e = cudaSuccess;
  if (st == EDP_OK) {
    std::memset(page, 1, bytes);  // fault the pages in before timing
    std::memset(pin, 2, bytes);
    e = cudaMemset(d, 3, 2 * bytes);
    uint8_t *pin_dev = nullptr;
    if (e == cudaSuccess) e = cudaHostGetDevicePointer((void **)&pin_dev, pin, 0);
    if (e == cudaSuccess)
      r.hbm_copy = best_gpu(bytes, [&] { cudaMemcpyAsync(d + bytes, d, bytes, cudaMemcpyDeviceToDevice, 0); }, &e);
    if (e == cudaSuccess)
      r.h2d_pinned = best_gpu(bytes, [&] { cudaMemcpyAsync(d, pin, bytes, cudaMemcpyHostToDevice, 0); }, &e);
    if (e == cudaSuccess)
      r.d2h_pinned = best_gpu(bytes, [&] { cudaMemcpyAsync(pin, d, bytes, cudaMemcpyDeviceToHost, 0); }, &e);
    if (e == cudaSuccess)
      r.h2d_pageable = best_gpu(bytes, [&] { cudaMemcpyAsync(d, page, bytes, cudaMemcpyHostToDevice, 0); }, &e);
    if (e == cudaSuccess)
      r.zero_copy_read = best_gpu(bytes, [&] { edp::launch_probe_read(pin_dev, bytes, fold, 0); }, &e);
    if (e == cudaSuccess) {
      for (int k = 0; k < 3; ++k) {
        const auto t0 = std::chrono::steady_clock::now();
        std::memcpy(pin, page, bytes);
        const double s = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
        if (s > 0.0 && bytes / s > r.host_copy) r.host_copy = bytes / s;
      }
    }
    if (e != cudaSuccess) st = EDP_ERR_CUDA;
  }
  cudaDeviceSynchronize();
  if (d) cudaFree(d);
  if (fold) cudaFree(fold);
  if (pin) cudaFreeHost(pin);
  std::free(page);
  cudaGetLastError();
  if (st == EDP_OK) *out = r;
  return st;
}

}  // extern "C"
