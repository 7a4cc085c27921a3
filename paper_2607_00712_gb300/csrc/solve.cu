// Closed-form absorption solve (Sec. 3.2, Eq. 5-6) in fp64 on the GPU.
//
//   M  = G + lambda I                      (G symmetrised from its upper tiles)
//   L  = chol(M)                           (right-looking blocked Cholesky, NB = 32)
//   Y  = L^{-1} (X W)                      (blocked forward substitution)
//   dW = L^{-T} Y                          (blocked back substitution)
//   eps = tr(W^T S W) - ||Y||_F^2 - lambda ||dW||_F^2
// The eps expression is Eq. 6 expanded with the normal equations
// (G + lambda I) dW = X W, which give tr(dW^T G dW) = ||Y||^2 - lambda||dW||^2
// and tr(dW^T X W) = ||Y||^2.  It runs once per layer at the transition, so
// the kernels are plain fp64 SIMT code bounded by GB300's fp64 rate.
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"

namespace ispa {

namespace {

constexpr int NB = 32;    // Cholesky / triangular block
constexpr int TB = 64;    // GEMM tile
constexpr int TK = 16;    // GEMM k step

enum MatMode : int { M_F32 = 0, M_F64 = 1, M_F64_T = 2, M_F32_SYM = 3 };

struct MatRef {
  const void* p;
  int64_t ld;
  int mode;
};

__device__ __forceinline__ double mat_get(const MatRef& m, int64_t i, int64_t k) {
  switch (m.mode) {
    case M_F32: return static_cast<double>(static_cast<const float*>(m.p)[i * m.ld + k]);
    case M_F64: return static_cast<const double*>(m.p)[i * m.ld + k];
    case M_F64_T: return static_cast<const double*>(m.p)[k * m.ld + i];
    default: {
      const int64_t a = i < k ? i : k, b = i < k ? k : i;
      return static_cast<double>(static_cast<const float*>(m.p)[a * m.ld + b]);
    }
  }
}

// C[M][N] = alpha * A[M][K] B[K][N] + beta * C (fp64).  lower_only skips tiles
// strictly above the diagonal of C.
__global__ void __launch_bounds__(256) dgemm_kernel(int M, int N, int K, MatRef A, MatRef B, double* C,
                                                    int64_t ldc, double alpha, double beta,
                                                    int lower_only) {
  const int bx = blockIdx.x, by = blockIdx.y;
  if (lower_only && bx * TB > by * TB + TB - 1) return;
  __shared__ double As[TK][TB + 1];
  __shared__ double Bs[TK][TB + 1];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  double acc[4][4] = {};
  const int row0 = by * TB, col0 = bx * TB;
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int e = threadIdx.x; e < TK * TB; e += 256) {
      const int kk = e / TB, ii = e % TB;
      const int gi = row0 + ii, gk = k0 + kk;
      As[kk][ii] = (gi < M && gk < K) ? mat_get(A, gi, gk) : 0.0;
      const int gj = col0 + ii;
      Bs[kk][ii] = (gk < K && gj < N) ? mat_get(B, gk, gj) : 0.0;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      double a[4], b[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) a[r] = As[kk][ty + 16 * r];
#pragma unroll
      for (int c = 0; c < 4; ++c) b[c] = Bs[kk][tx + 16 * c];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fma(a[r], b[c], acc[r][c]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int gi = row0 + ty + 16 * r;
    if (gi >= M) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int gj = col0 + tx + 16 * c;
      if (gj >= N) continue;
      double* cp = C + gi * ldc + gj;
      *cp = alpha * acc[r][c] + (beta == 0.0 ? 0.0 : beta * *cp);
    }
  }
}

// M = sym(G) + lambda I, fp64 [D][D].  G's upper triangle is always valid.
__global__ void form_spd_kernel(const float* __restrict__ gram, int D, double lambda, double* __restrict__ L) {
  const int64_t n = static_cast<int64_t>(D) * D;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(e / D), j = static_cast<int>(e % D);
    const int a = i < j ? i : j, b = i < j ? j : i;
    double v = static_cast<double>(gram[static_cast<int64_t>(a) * (2 * D) + b]);
    if (i == j) v += lambda;
    L[e] = v;
  }
}

// Unblocked Cholesky of the nb x nb diagonal block at (k0, k0), in place (lower).
__global__ void __launch_bounds__(256) potrf_diag_kernel(double* L, int D, int k0, int nb, int* flag) {
  __shared__ double a[NB][NB + 1];
  for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
    const int i = e / nb, j = e % nb;
    a[i][j] = L[static_cast<int64_t>(k0 + i) * D + k0 + j];
  }
  __syncthreads();
  for (int j = 0; j < nb; ++j) {
    if (threadIdx.x == 0) {
      double d = a[j][j];
      if (!(d > 0.0)) {
        atomicExch(flag, 1);
        d = 1.0;  // keep the remaining arithmetic finite; the caller reports NOT_SPD
      }
      a[j][j] = sqrt(d);
    }
    __syncthreads();
    for (int i = j + 1 + threadIdx.x; i < nb; i += blockDim.x) a[i][j] /= a[j][j];
    __syncthreads();
    const int m = nb - j - 1;
    for (int e = threadIdx.x; e < m * m; e += blockDim.x) {
      const int i = j + 1 + e / m, k = j + 1 + e % m;
      if (k <= i) a[i][k] -= a[i][j] * a[k][j];
    }
    __syncthreads();
  }
  for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
    const int i = e / nb, j = e % nb;
    L[static_cast<int64_t>(k0 + i) * D + k0 + j] = j <= i ? a[i][j] : 0.0;
  }
}

// Panel: rows i >= k0+nb solve x L11^T = a (one row per thread).
__global__ void __launch_bounds__(128) trsm_panel_kernel(double* L, int D, int k0, int nb) {
  __shared__ double l11[NB][NB + 1];
  for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
    const int i = e / nb, j = e % nb;
    l11[i][j] = L[static_cast<int64_t>(k0 + i) * D + k0 + j];
  }
  __syncthreads();
  const int i = k0 + nb + blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= D) return;
  double* row = L + static_cast<int64_t>(i) * D + k0;
  double x[NB];
#pragma unroll
  for (int j = 0; j < NB; ++j) {
    if (j < nb) {
      double v = row[j];
      for (int m = 0; m < j; ++m) v -= x[m] * l11[j][m];
      x[j] = v / l11[j][j];
    }
  }
#pragma unroll
  for (int j = 0; j < NB; ++j)
    if (j < nb) row[j] = x[j];
}

// Forward block: L11 Y1 = B1 for rows k0..k0+nb (one column of B per thread).
__global__ void trsv_fwd_kernel(const double* L, int D, int k0, int nb, double* B, int n_cols) {
  __shared__ double l11[NB][NB + 1];
  for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
    const int i = e / nb, j = e % nb;
    l11[i][j] = L[static_cast<int64_t>(k0 + i) * D + k0 + j];
  }
  __syncthreads();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n_cols) return;
  double y[NB];
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    if (i < nb) {
      double v = B[static_cast<int64_t>(k0 + i) * n_cols + c];
      for (int m = 0; m < i; ++m) v -= l11[i][m] * y[m];
      y[i] = v / l11[i][i];
      B[static_cast<int64_t>(k0 + i) * n_cols + c] = y[i];
    }
  }
}

// Backward block: L11^T Z1 = Y1 for rows k0..k0+nb.
__global__ void trsv_bwd_kernel(const double* L, int D, int k0, int nb, double* B, int n_cols) {
  __shared__ double l11[NB][NB + 1];
  for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
    const int i = e / nb, j = e % nb;
    l11[i][j] = L[static_cast<int64_t>(k0 + i) * D + k0 + j];
  }
  __syncthreads();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n_cols) return;
  double z[NB];
#pragma unroll
  for (int i = NB - 1; i >= 0; --i) {
    if (i < nb) {
      double v = B[static_cast<int64_t>(k0 + i) * n_cols + c];
      for (int m = i + 1; m < nb; ++m) v -= l11[m][i] * z[m];
      z[i] = v / l11[i][i];
      B[static_cast<int64_t>(k0 + i) * n_cols + c] = z[i];
    }
  }
}

// out += sum_e x[e] * y[e]  (y of type float or double; y == nullptr means y = x)
template <typename TY>
__global__ void __launch_bounds__(256) dot_kernel(const double* __restrict__ x, const TY* __restrict__ y,
                                                  int64_t n, double* out) {
  double s = 0.0;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x)
    s += x[e] * (y ? static_cast<double>(y[e]) : x[e]);
  __shared__ double red[8];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    s = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (threadIdx.x == 0) atomicAdd(out, s);
  }
}

__global__ void to_f32_kernel(const double* __restrict__ x, float* __restrict__ y, int64_t n) {
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x)
    y[e] = static_cast<float>(x[e]);
}

size_t align256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

struct SolveWs {
  double* L;
  double* B;
  double* SW;
  double* scal;  // [0] ||Y||^2, [1] ||dW||^2, [2] <W, S W>
  int* flag;
};

SolveWs carve(void* ws, int D, int d_out) {
  uint8_t* p = static_cast<uint8_t*>(ws);
  SolveWs w;
  w.L = reinterpret_cast<double*>(p);
  p += align256(static_cast<size_t>(D) * D * 8);
  w.B = reinterpret_cast<double*>(p);
  p += align256(static_cast<size_t>(D) * d_out * 8);
  w.SW = reinterpret_cast<double*>(p);
  p += align256(static_cast<size_t>(D) * d_out * 8);
  w.scal = reinterpret_cast<double*>(p);
  p += 256;
  w.flag = reinterpret_cast<int*>(p);
  return w;
}

cudaError_t gemm(int M, int N, int K, MatRef A, MatRef B, double* C, int64_t ldc, double alpha,
                 double beta, bool lower_only, cudaStream_t s) {
  if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
  dim3 grid((N + TB - 1) / TB, (M + TB - 1) / TB);
  dgemm_kernel<<<grid, 256, 0, s>>>(M, N, K, A, B, C, ldc, alpha, beta, lower_only ? 1 : 0);
  return cudaGetLastError();
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  if (b > 152 * 16) b = 152 * 16;
  return static_cast<int>(b < 1 ? 1 : b);
}

}  // namespace

size_t ls_solve_ws_bytes(int32_t D, int32_t d_out) {
  return align256(static_cast<size_t>(D) * D * 8) + 2 * align256(static_cast<size_t>(D) * d_out * 8) + 512;
}

ispa_status run_ls_solve(int32_t D, const float* gram, const float* W, int32_t d_out, double lambda,
                         float* dW, double* eps_out, void* ws, cudaStream_t s) {
  SolveWs w = carve(ws, D, d_out);
  const int64_t ldg = 2 * static_cast<int64_t>(D);
  const int64_t nDo = static_cast<int64_t>(D) * d_out;
#define ISPA_CK(x)                            \
  do {                                        \
    if ((x) != cudaSuccess) return ISPA_ERR_CUDA; \
  } while (0)
  ISPA_CK(cudaMemsetAsync(w.scal, 0, 256 + sizeof(int), s));
  form_spd_kernel<<<grid_for(static_cast<int64_t>(D) * D, 256), 256, 0, s>>>(gram, D, lambda, w.L);
  ISPA_CK(cudaGetLastError());
  // Cholesky, right-looking
  for (int k0 = 0; k0 < D; k0 += NB) {
    const int nb = D - k0 < NB ? D - k0 : NB;
    potrf_diag_kernel<<<1, 256, 0, s>>>(w.L, D, k0, nb, w.flag);
    ISPA_CK(cudaGetLastError());
    const int rest = D - k0 - nb;
    if (rest > 0) {
      trsm_panel_kernel<<<(rest + 127) / 128, 128, 0, s>>>(w.L, D, k0, nb);
      ISPA_CK(cudaGetLastError());
      double* L22 = w.L + static_cast<int64_t>(k0 + nb) * D + (k0 + nb);
      const double* L21 = w.L + static_cast<int64_t>(k0 + nb) * D + k0;
      ISPA_CK(gemm(rest, rest, nb, MatRef{L21, D, M_F64}, MatRef{L21, D, M_F64_T}, L22, D, -1.0, 1.0,
                   true, s));
    }
  }
  // B = X W
  ISPA_CK(gemm(D, d_out, D, MatRef{gram + D, ldg, M_F32}, MatRef{W, d_out, M_F32}, w.B, d_out, 1.0, 0.0,
               false, s));
  // forward substitution
  for (int k0 = 0; k0 < D; k0 += NB) {
    const int nb = D - k0 < NB ? D - k0 : NB;
    trsv_fwd_kernel<<<(d_out + 127) / 128, 128, 0, s>>>(w.L, D, k0, nb, w.B, d_out);
    ISPA_CK(cudaGetLastError());
    const int rest = D - k0 - nb;
    if (rest > 0)
      ISPA_CK(gemm(rest, d_out, nb, MatRef{w.L + static_cast<int64_t>(k0 + nb) * D + k0, D, M_F64},
                   MatRef{w.B + static_cast<int64_t>(k0) * d_out, d_out, M_F64},
                   w.B + static_cast<int64_t>(k0 + nb) * d_out, d_out, -1.0, 1.0, false, s));
  }
  dot_kernel<double><<<grid_for(nDo, 256), 256, 0, s>>>(w.B, nullptr, nDo, w.scal + 0);
  ISPA_CK(cudaGetLastError());
  // back substitution
  const int last = ((D - 1) / NB) * NB;
  for (int k0 = last; k0 >= 0; k0 -= NB) {
    const int nb = D - k0 < NB ? D - k0 : NB;
    trsv_bwd_kernel<<<(d_out + 127) / 128, 128, 0, s>>>(w.L, D, k0, nb, w.B, d_out);
    ISPA_CK(cudaGetLastError());
    if (k0 > 0)
      ISPA_CK(gemm(k0, d_out, nb, MatRef{w.L + static_cast<int64_t>(k0) * D, D, M_F64_T},
                   MatRef{w.B + static_cast<int64_t>(k0) * d_out, d_out, M_F64}, w.B, d_out, -1.0, 1.0,
                   false, s));
  }
  dot_kernel<double><<<grid_for(nDo, 256), 256, 0, s>>>(w.B, nullptr, nDo, w.scal + 1);
  ISPA_CK(cudaGetLastError());
  to_f32_kernel<<<grid_for(nDo, 256), 256, 0, s>>>(w.B, dW, nDo);
  ISPA_CK(cudaGetLastError());
  // <W, S W>
  ISPA_CK(gemm(D, d_out, D, MatRef{gram + static_cast<int64_t>(D) * ldg + D, ldg, M_F32_SYM},
               MatRef{W, d_out, M_F32}, w.SW, d_out, 1.0, 0.0, false, s));
  dot_kernel<float><<<grid_for(nDo, 256), 256, 0, s>>>(w.SW, W, nDo, w.scal + 2);
  ISPA_CK(cudaGetLastError());
  double scal[3];
  int flag = 0;
  ISPA_CK(cudaMemcpyAsync(scal, w.scal, sizeof(scal), cudaMemcpyDeviceToHost, s));
  ISPA_CK(cudaMemcpyAsync(&flag, w.flag, sizeof(int), cudaMemcpyDeviceToHost, s));
  ISPA_CK(cudaStreamSynchronize(s));
#undef ISPA_CK
  if (eps_out) *eps_out = scal[2] - scal[0] - lambda * scal[1];
  return flag ? ISPA_ERR_NOT_SPD : ISPA_OK;
}

}  // namespace ispa
