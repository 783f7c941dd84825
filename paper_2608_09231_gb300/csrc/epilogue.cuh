// Fused GEMM epilogues: every projection of the DiT block finishes here, so that no
// separate elementwise pass re-reads its output.
//   QKV (+ RoPE on q and k, V written transposed per head for the attention kernel's
//   K-major B operand) and the GELU'd MLP half of a single-stream block's linear1,
//   gated residual h += g * y (out-projection, linear2, MLP down), plain/GELU/SiLU
//   stores, and the flow-matching Euler update x += (sigma_{t+1} - sigma_t) v.
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace bag {

BAG_DEV int epi_step(const Epi& e) { return e.st ? e.st->t : 0; }

// Early exit for kernels captured on one side of the full/reuse branch.
BAG_DEV bool epi_skip(const DevState* st, int flag_want) {
  return st != nullptr && flag_want >= 0 && st->flag != flag_want;
}

// type: kStoreF32, kStoreBF16 or kStoreF16
template <int NV>
BAG_DEV void store_vals(void* base, long idx, const float* v, int type) {
  if (type == kStoreF16) {
    __half* p = reinterpret_cast<__half*>(base) + idx;
    if constexpr (NV % 8 == 0) {
      if ((reinterpret_cast<uintptr_t>(p) & 15) == 0) {
#pragma unroll
        for (int j = 0; j < NV; j += 8) {
          uint4 u;
          u.x = pack_f16x2(v[j], v[j + 1]);
          u.y = pack_f16x2(v[j + 2], v[j + 3]);
          u.z = pack_f16x2(v[j + 4], v[j + 5]);
          u.w = pack_f16x2(v[j + 6], v[j + 7]);
          *reinterpret_cast<uint4*>(p + j) = u;
        }
        return;
      }
    }
#pragma unroll
    for (int j = 0; j < NV; ++j) p[j] = __float2half_rn(v[j]);
  } else if (type == kStoreBF16) {
    __nv_bfloat16* p = reinterpret_cast<__nv_bfloat16*>(base) + idx;
    if constexpr (NV % 8 == 0) {
      if ((reinterpret_cast<uintptr_t>(p) & 15) == 0) {
#pragma unroll
        for (int j = 0; j < NV; j += 8) {
          uint4 u;
          u.x = pack_bf16x2(v[j], v[j + 1]);
          u.y = pack_bf16x2(v[j + 2], v[j + 3]);
          u.z = pack_bf16x2(v[j + 4], v[j + 5]);
          u.w = pack_bf16x2(v[j + 6], v[j + 7]);
          *reinterpret_cast<uint4*>(p + j) = u;
        }
        return;
      }
    }
#pragma unroll
    for (int j = 0; j < NV; ++j) p[j] = __float2bfloat16_rn(v[j]);
  } else {
    float* p = reinterpret_cast<float*>(base) + idx;
    if constexpr (NV % 4 == 0) {
      if ((reinterpret_cast<uintptr_t>(p) & 15) == 0) {
#pragma unroll
        for (int j = 0; j < NV; j += 4)
          *reinterpret_cast<float4*>(p + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        return;
      }
    }
#pragma unroll
    for (int j = 0; j < NV; ++j) p[j] = v[j];
  }
}

// Apply the epilogue to NV consecutive accumulators v[0..NV) of output row `row`,
// columns [col0, col0 + NV).  NV is even and col0 is a multiple of NV; the chunk never
// straddles a q/k/v/mlp boundary (those are multiples of 64 columns).
// Bias of the output columns col0 .. col0 + NV - 1 (16-byte loads when aligned).
template <int NV>
BAG_DEV void epi_add_bias(const Epi& e, int col0, float* v) {
  if (e.bias) {
    if (NV % 4 == 0 && (reinterpret_cast<uintptr_t>(e.bias + col0) & 15) == 0) {
      const float4* b4 = reinterpret_cast<const float4*>(e.bias + col0);
#pragma unroll
      for (int j = 0; j < NV; j += 4) {
        const float4 b = __ldg(b4 + j / 4);
        v[j] += b.x;
        v[j + 1] += b.y;
        v[j + 2] += b.z;
        v[j + 3] += b.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < NV; ++j) v[j] += __ldg(e.bias + col0 + j);
    }
  }
}

// EPI_QKV q / k columns (region 0 / 1): per-head RMSNorm (when the block has it), then
// the rotation of joint-sequence row jr; cc is the column within the region.
template <int NV>
BAG_DEV void epi_qk_transform(const Epi& e, int jr, int cc, int region, float* v, float rs) {
  if (region < 2 && e.qn_q) {  // per-head RMSNorm of q and k, before the rotation
    const float* w = (region == 0 ? e.qn_q : e.qn_k) + cc % e.dh;
#pragma unroll
    for (int j = 0; j < NV; ++j) v[j] = v[j] * rs * __ldg(w + j);
  }
  if (region < 2 && e.rope) {
    const int e0 = cc % e.dh;
    const float2* cs = e.rope + (long)jr * (e.dh / 2) + e0 / 2;
    if constexpr (NV % 4 == 0) {
      // two (cos, sin) pairs per 16-byte load (the table row offset is a multiple of
      // NV / 2 pairs, so 16-byte aligned)
      const float4* cs4 = reinterpret_cast<const float4*>(cs);
#pragma unroll
      for (int p = 0; p < NV / 4; ++p) {
        const float4 r = __ldg(cs4 + p);
        const float x0 = v[4 * p], x1 = v[4 * p + 1], x2 = v[4 * p + 2], x3 = v[4 * p + 3];
        v[4 * p] = x0 * r.x - x1 * r.y;
        v[4 * p + 1] = x0 * r.y + x1 * r.x;
        v[4 * p + 2] = x2 * r.z - x3 * r.w;
        v[4 * p + 3] = x2 * r.w + x3 * r.z;
      }
    } else {
#pragma unroll
      for (int p = 0; p < NV / 2; ++p) {
        const float2 r = __ldg(cs + p);
        const float x0 = v[2 * p], x1 = v[2 * p + 1];
        v[2 * p] = x0 * r.x - x1 * r.y;
        v[2 * p + 1] = x0 * r.y + x1 * r.x;
      }
    }
  }
}

// rs: EPI_QKV with QK-norm, 1 / RMS of the head that columns col0 .. col0 + NV - 1 of
// this row belong to (computed by the caller over the whole head).
template <int NV>
BAG_DEV void epi_apply(const Epi& e, int t, int row, int col0, float* v, float rs = 1.f) {
  if (row >= e.M || col0 >= e.N) return;
  epi_add_bias<NV>(e, col0, v);
  switch (e.kind) {
    case EPI_STORE:
      store_vals<NV>(e.out, (long)row * e.ldo + col0, v, e.out_bf16);
      break;
    case EPI_GELU:
      if (e.out_bf16) {
#pragma unroll
        for (int j = 0; j < NV; ++j) v[j] = gelu_tanh_fast(v[j]);
      } else {
#pragma unroll
        for (int j = 0; j < NV; ++j) v[j] = gelu_tanh(v[j]);
      }
      store_vals<NV>(e.out, (long)row * e.ldo + col0, v, e.out_bf16);
      break;
    case EPI_SILU:
#pragma unroll
      for (int j = 0; j < NV; ++j) v[j] = silu(v[j]);
      store_vals<NV>(e.out, (long)row * e.ldo + col0, v, e.out_bf16);
      break;
    case EPI_QKV: {
      const int lc = col0 + e.col_base;
      const int region = lc / e.d;
      if (region >= 3) {
#pragma unroll
        for (int j = 0; j < NV; ++j) v[j] = e.act_bf16 ? gelu_tanh_fast(v[j]) : gelu_tanh(v[j]);
        store_vals<NV>(e.mlp, (long)row * e.ldm + (lc - 3 * e.d), v, e.act_bf16);
        break;
      }
      const bool br1 = e.br_rows > 0 && row >= e.br_rows;       // unconditional branch
      const int jr = row - (br1 ? e.br_rows : 0) + e.row_off;  // joint-sequence row
      const long qr = jr + (br1 ? e.br_qk : 0);                // q / k / v buffer row
      const int cc = lc - region * e.d;
      if (region < 2) epi_qk_transform<NV>(e, jr, cc, region, v, rs);
      if (region == 0) {
        store_vals<NV>(e.q, qr * e.ldqk + cc, v, e.qkv_type);
      } else if (region == 1) {
        store_vals<NV>(e.k, qr * e.ldqk + cc, v, e.qkv_type);
      } else if (e.v_mode == 0) {
        store_vals<NV>(e.v, qr * e.ldqk + cc, v, e.qkv_type);
      } else {
        // transposed per head: vt[(head * dh + e) * vpad + token]
        if (e.qkv_type == kStoreF16) {
          __half* vt = reinterpret_cast<__half*>(e.v) + (br1 ? e.br_vt : 0);
#pragma unroll
          for (int j = 0; j < NV; ++j) vt[(long)(cc + j) * e.vpad + jr] = __float2half_rn(v[j]);
        } else if (e.qkv_type == kStoreBF16) {
          __nv_bfloat16* vt = reinterpret_cast<__nv_bfloat16*>(e.v) + (br1 ? e.br_vt : 0);
#pragma unroll
          for (int j = 0; j < NV; ++j) vt[(long)(cc + j) * e.vpad + jr] = __float2bfloat16_rn(v[j]);
        } else {
          float* vt = reinterpret_cast<float*>(e.v) + (br1 ? e.br_vt : 0);
#pragma unroll
          for (int j = 0; j < NV; ++j) vt[(long)(cc + j) * e.vpad + jr] = v[j];
        }
      }
      break;
    }
    case EPI_GATED_RES: {
      const float* g = (e.br_rows > 0 && row >= e.br_rows ? e.gate_u : e.gate) + (long)t * e.gate_step + col0;
      float* r = e.resid + (long)row * e.ldr + col0;
      if (NV % 4 == 0 && ((reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(r)) & 15) == 0) {
#pragma unroll
        for (int j = 0; j < NV; j += 4) {
          const float4 g4 = __ldg(reinterpret_cast<const float4*>(g + j));
          float4 h = *reinterpret_cast<float4*>(r + j);
          h.x += g4.x * v[j];
          h.y += g4.y * v[j + 1];
          h.z += g4.z * v[j + 2];
          h.w += g4.w * v[j + 3];
          *reinterpret_cast<float4*>(r + j) = h;
        }
      } else {
#pragma unroll
        for (int j = 0; j < NV; ++j) r[j] += __ldg(g + j) * v[j];
      }
      break;
    }
    case EPI_RES_ADD: {
      float* r = e.resid + (long)row * e.ldr + col0;
#pragma unroll
      for (int j = 0; j < NV; ++j) r[j] += v[j];
      break;
    }
    case EPI_EULER: {
      const float ds = e.dsig[t];
      float* x = e.x + (long)row * e.ldx + col0;
      if (e.vcond) {  // classifier-free guidance: v_u + g (v_c - v_u)
        const float* vc = e.vcond + (long)row * e.ldx + col0;
#pragma unroll
        for (int j = 0; j < NV; ++j) v[j] = v[j] + e.guidance * (vc[j] - v[j]);
      }
      float nx[NV];
      if (e.uni_coef) {
        // UniPC: m_i = x_i - sigma_i v; corrected x_i^c (a combination of x_i, the previous
        // corrected sample and m_{i-1}, m_{i-2}, m_i); x_{i+1} from x_i^c, m_i, m_{i-1}.
        // Terms whose weight is zero are not read (uniform across the grid).
        const float* k = e.uni_coef + (long)t * kUniCoefs;
        const long idx = (long)row * e.ldx + col0;
        float* mcur = (t & 1) ? e.uni_m1 : e.uni_m0;        // holds m_{i-2}; receives m_i
        const float* mprev = (t & 1) ? e.uni_m0 : e.uni_m1;  // m_{i-1}
        float* xl = e.uni_xl + idx;
        const bool use_last = k[UC_CLAST] != 0.f, use_m2 = k[UC_CM2] != 0.f;
        const bool use_m1 = k[UC_CM1] != 0.f || k[UC_DM1] != 0.f;
#pragma unroll
        for (int j = 0; j < NV; ++j) {
          const float m = x[j] - k[UC_SIG] * v[j];
          float xc = k[UC_CX] * x[j] + k[UC_CMT] * m;
          const float m1 = use_m1 ? mprev[idx + j] : 0.f;
          if (use_last) xc += k[UC_CLAST] * xl[j];
          if (use_m1) xc += k[UC_CM1] * m1;
          if (use_m2) xc += k[UC_CM2] * mcur[idx + j];
          nx[j] = k[UC_DX] * xc + k[UC_DM0] * m + k[UC_DM1] * m1;
          xl[j] = xc;
          mcur[idx + j] = m;
          x[j] = nx[j];
        }
      } else {
#pragma unroll
        for (int j = 0; j < NV; ++j) {
          nx[j] = x[j] + ds * v[j];
          x[j] = nx[j];
        }
      }
      if (e.xb) {
        // next step's patch-embedding operand: bf16 hi | lo halves of the new latent
        float lo[NV];
#pragma unroll
        for (int j = 0; j < NV; ++j) lo[j] = nx[j] - bf16_round(nx[j]);
        store_vals<NV>(e.xb, (long)row * 2 * e.ldx + col0, nx, kStoreBF16);
        store_vals<NV>(e.xb, (long)row * 2 * e.ldx + e.ldx + col0, lo, kStoreBF16);
      }
      break;
    }
    case EPI_VEC: {
#pragma unroll
      for (int j = 0; j < NV; ++j) v[j] += (e.addend ? e.addend[col0 + j] : 0.f);
      store_vals<NV>(e.out, (long)row * e.ldo + col0, v, 0);
#pragma unroll
      for (int j = 0; j < NV; ++j) v[j] = silu(v[j]);
      store_vals<NV>(e.out2, (long)row * e.ldo2 + col0, v, e.out2_bf16);
      break;
    }
    case EPI_DUAL_F32:
      store_vals<NV>(e.out, (long)row * e.ldo + col0, v, 0);
      store_vals<NV>(e.out2, (long)row * e.ldo2 + col0, v, 0);
      break;
    default:
      break;
  }
}

}  // namespace bag
