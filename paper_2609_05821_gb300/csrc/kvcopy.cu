// Index-driven gather / scatter of selected K/V rows for the selective
// recompute (Conduit Sec. 3.1 and 3.5): rows[l][i][g][:] <-> cache[l][g][idx_i][:],
// all layers, both K and V, contiguous or paged, in one launch. Each thread
// moves one 16-byte chunk of K and the matching chunk of V; the exchange
// mode reads the stale chunk out and then writes the fresh one in its place.
#include "internal.cuh"

namespace conduit {
namespace {

template <int kMode>  // 0 gather, 1 scatter, 2 exchange
__global__ void __launch_bounds__(256) kv_copy_kernel(KvDev kv, BatchDev b, const int32_t* idx,
                                                      const int32_t* idx_off, int32_t n_sel,
                                                      int esize, char* k_rows, char* v_rows,
                                                      const char* k_new, const char* v_new) {
  const int r = blockIdx.y, l = blockIdx.z;
  const int i0 = idx_off[r], k_r = idx_off[r + 1] - i0;
  const int cpr = kv.d * esize / 16;  // chunks per head row
  const int64_t lin = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (lin >= int64_t(k_r) * kv.Hkv * cpr) return;
  const int il = int(lin / (kv.Hkv * cpr));
  const int rem = int(lin % (kv.Hkv * cpr));
  const int g = rem / cpr, c = rem % cpr;
  const int i = i0 + il;
  const int t = idx[i];
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  if (t < 0 || t >= N) return;  // out-of-range indices are skipped
  const int64_t cache_off = kv.row(l, g, r, int64_t(t0) + t, t) * esize + int64_t(c) * 16;
  const int64_t rows_off = ((int64_t(l) * n_sel + i) * kv.Hkv + g) * int64_t(kv.d) * esize + c * 16;
  char* kc = static_cast<char*>(kv.k) + cache_off;
  char* vc = static_cast<char*>(kv.v) + cache_off;
  if (kMode == 1) {
    *reinterpret_cast<uint4*>(kc) = *reinterpret_cast<const uint4*>(k_rows + rows_off);
    *reinterpret_cast<uint4*>(vc) = *reinterpret_cast<const uint4*>(v_rows + rows_off);
  } else if (kMode == 0) {
    *reinterpret_cast<uint4*>(k_rows + rows_off) = *reinterpret_cast<const uint4*>(kc);
    *reinterpret_cast<uint4*>(v_rows + rows_off) = *reinterpret_cast<const uint4*>(vc);
  } else {
    const uint4 ko = *reinterpret_cast<const uint4*>(kc);
    const uint4 vo = *reinterpret_cast<const uint4*>(vc);
    const uint4 kn = *reinterpret_cast<const uint4*>(k_new + rows_off);
    const uint4 vn = *reinterpret_cast<const uint4*>(v_new + rows_off);
    *reinterpret_cast<uint4*>(k_rows + rows_off) = ko;
    *reinterpret_cast<uint4*>(v_rows + rows_off) = vo;
    *reinterpret_cast<uint4*>(kc) = kn;
    *reinterpret_cast<uint4*>(vc) = vn;
  }
}

}  // namespace

cudaError_t launch_kv_copy(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                           const int32_t* idx_off_dev, int32_t n_sel, int max_sel, int mode,
                           void* k_rows, void* v_rows, const void* k_new, const void* v_new,
                           cudaStream_t stream) {
  if (n_sel == 0 || max_sel == 0) return cudaSuccess;
  const int esize = kv.dtype == CONDUIT_BF16 ? 2 : 4;
  const int64_t per_req = int64_t(max_sel) * kv.Hkv * (kv.d * esize / 16);
  const dim3 grid(unsigned((per_req + 255) / 256), b.R, kv.L);
  char* kr = static_cast<char*>(k_rows);
  char* vr = static_cast<char*>(v_rows);
  const char* kn = static_cast<const char*>(k_new);
  const char* vn = static_cast<const char*>(v_new);
  if (mode == 1)
    kv_copy_kernel<1><<<grid, 256, 0, stream>>>(kv, b, idx, idx_off_dev, n_sel, esize, kr, vr, kn, vn);
  else if (mode == 0)
    kv_copy_kernel<0><<<grid, 256, 0, stream>>>(kv, b, idx, idx_off_dev, n_sel, esize, kr, vr, kn, vn);
  else
    kv_copy_kernel<2><<<grid, 256, 0, stream>>>(kv, b, idx, idx_off_dev, n_sel, esize, kr, vr, kn, vn);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
