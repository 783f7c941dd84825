// Joint attention softmax(q k^T / sqrt(dh)) v per head, flash-style (online softmax,
// O(N) memory).  This file holds the CUDA-core kernel used for the fp32
// configuration and for shapes the tensor-core kernel does not tile; the tcgen05
// kernel lives in attn_tc.cu.
#include <cmath>

#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace bag {

template <typename T>
BAG_DEV float ldv(const void* p, long i) {
  if constexpr (sizeof(T) == 2)
    return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(p)[i]);
  else
    return reinterpret_cast<const float*>(p)[i];
}

// CTA = 4 warps = 16 queries of one head; each warp owns 4 queries.  Key tiles of 32
// are staged in shared memory (K transposed so that lane j reads key j's column).
template <typename T, int DH>
__global__ void __launch_bounds__(128) attn_simt_kernel(const AttnArgs a) {
  grid_dep_sync();
  if (epi_skip(a.st, a.flag_want)) return;
  constexpr int QPW = 4, QPB = 16, KT = 32, R = DH / 32;
  __shared__ float Qs[QPB][DH];
  __shared__ float Kt[DH][KT + 1];
  __shared__ float Vs[KT][DH];
  const int head = blockIdx.y, q0 = blockIdx.x * QPB;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const float scale = rsqrtf((float)DH);
  for (int i = threadIdx.x; i < QPB * DH; i += blockDim.x) {
    const int r = i / DH, c = i % DH, q = q0 + r;
    Qs[r][c] = q < a.nq ? ldv<T>(a.q, (long)q * a.ldq + head * DH + c) * scale : 0.f;
  }
  float m[QPW], l[QPW], o[QPW][R];
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) o[i][r] = 0.f;
  }
  for (int kb = 0; kb < a.nk; kb += KT) {
    __syncthreads();
    for (int i = threadIdx.x; i < KT * DH; i += blockDim.x) {
      const int j = i / DH, c = i % DH, kk = kb + j;
      float kv = 0.f, vv = 0.f;
      if (kk < a.nk) {
        kv = ldv<T>(a.k, (long)kk * a.ldk + head * DH + c);
        vv = a.v_mode == 0 ? ldv<T>(a.v, (long)kk * a.ldv + head * DH + c)
                           : ldv<T>(a.v, (long)(head * DH + c) * a.vpad + kk);
      }
      Kt[c][j] = kv;
      Vs[j][c] = vv;
    }
    __syncthreads();
    const bool valid = kb + lane < a.nk;
#pragma unroll
    for (int qi = 0; qi < QPW; ++qi) {
      const int qr = warp * QPW + qi;
      float s = 0.f;
#pragma unroll 8
      for (int c = 0; c < DH; ++c) s += Qs[qr][c] * Kt[c][lane];
      s = valid ? s : -INFINITY;
      float mx = s;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float mn = fmaxf(m[qi], mx);
      const float p = valid ? expf(s - mn) : 0.f;
      const float corr = expf(m[qi] - mn);
      float ps = p;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
      l[qi] = l[qi] * corr + ps;
#pragma unroll
      for (int r = 0; r < R; ++r) o[qi][r] *= corr;
      for (int j = 0; j < KT; ++j) {
        const float pj = __shfl_sync(0xffffffffu, p, j);
#pragma unroll
        for (int r = 0; r < R; ++r) o[qi][r] += pj * Vs[j][lane + 32 * r];
      }
      m[qi] = mn;
    }
  }
#pragma unroll
  for (int qi = 0; qi < QPW; ++qi) {
    const int q = q0 + warp * QPW + qi;
    if (q >= a.nq) continue;
    const float inv = 1.f / l[qi];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const long idx = (long)q * a.ldo + head * DH + lane + 32 * r;
      const float val = o[qi][r] * inv;
      void* ob = (a.o2 && q >= a.o_split) ? a.o2 : a.o;
      if (a.bf16)
        reinterpret_cast<__nv_bfloat16*>(ob)[idx] = __float2bfloat16_rn(val);
      else
        reinterpret_cast<float*>(ob)[idx] = val;
    }
  }
}

cudaError_t attention_tc(const AttnArgs& a, int* err, cudaStream_t s);

cudaError_t attention(const AttnArgs& a, int* err, cudaStream_t s, int force_simt) {
  if (a.nq <= 0) return cudaSuccess;
  // bf16 attention runs on the tensor cores; a call the tensor-core kernel cannot take
  // (head_dim != 128, V not transposed, unaligned operands) is refused rather than sent
  // to the CUDA-core kernel, which serves fp32 backbones and explicit cross-checks only
  if (a.bf16 && !force_simt) {
    if (!attention_tc_supported(a)) return cudaErrorNotSupported;
    return attention_tc(a, err, s);
  }
  if (a.f16 || a.nbr > 1) return cudaErrorNotSupported;  // tensor-core kernel only
  dim3 grid((a.nq + 15) / 16, a.heads);
  if (a.dh == 64) {
    if (a.bf16)
      launch_kernel(attn_simt_kernel<__nv_bfloat16, 64>, grid, 128, 0, s, a);
    else
      launch_kernel(attn_simt_kernel<float, 64>, grid, 128, 0, s, a);
  } else if (a.dh == 128) {
    if (a.bf16)
      launch_kernel(attn_simt_kernel<__nv_bfloat16, 128>, grid, 128, 0, s, a);
    else
      launch_kernel(attn_simt_kernel<float, 128>, grid, 128, 0, s, a);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace bag
