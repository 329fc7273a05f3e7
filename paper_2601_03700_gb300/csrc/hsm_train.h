// Launchers of the HSM training-step kernels (hsm_train.cu).  Rows are dense: row r of every
// [n, C] buffer is example r; T is the model dtype (dt = 1: bf16, else fp32).
#pragma once
#include "common.cuh"

namespace adept {

// One column sum: out[c] = sum_r A[r][c] (* B[r][c]) (* rs[r]), A and B [n][C] row-major.
struct ColJob {
  const float* A;
  const float* B;
  const float* rs;
  int C;
  float* out;
};
constexpr int HT_COLSUM_MAX_JOBS = 4;
constexpr int HT_COLSUM_ROWS = 32;   // rows per partial sum
struct ColJobs {
  ColJob j[HT_COLSUM_MAX_JOBS];
  int nj;
  int n;
  int rows_per;                       // set by the launcher
  int cb[HT_COLSUM_MAX_JOBS + 1];     // first column block of each job (launcher)
  int pc[HT_COLSUM_MAX_JOBS + 1];     // first partial column of each job (launcher)
};
// Partial-sum columns a job group needs: chunks(n) * sum of C.
int ht_colsum_chunks(int n);

// One AdamW parameter segment: rows x cols fp32 values at theta/grad/m/v + off; optional
// copies of the updated values: wf fp32 [rows][cols], wt T [rows][cols], wT T [cols][rows].
struct AdamSeg {
  long long off;
  int rows, cols;
  float* wf;
  void* wt;
  void* wT;
  int tile0, tiles_x;   // set by the launcher
};
constexpr int HT_MAX_SEGS = 12;
struct AdamArgs {
  float* theta;
  const float* grad;
  float* m;
  float* v;
  float lr, b1, b2, eps, wd;
  float ibc1, ibc2;   // 1 / (1 - b1^t), 1 / (1 - b2^t)
  int nseg;
  AdamSeg seg[HT_MAX_SEGS];
};

// Cross-entropy rows (logits [n][ldl], V used) -> lossr[n], gradient dl [n][Vp] (T); loss
// (optional, device scalar) = mean of lossr.
void ht_launch_ce(cudaStream_t st, int dt, const float* logits, int ldl, int n, int V, int Vp, const int* target,
                  float* lossr, void* dl, float* loss, unsigned* err);
// Encoder step (Sec. 4.3): similarity rows (lossr[n] = 1 - cos, dxh [n][D] overwritten),
// classifier rows (zp [n_cls][D] pooler pre-activations -> lossc[n_cls], dpt [n_cls][D] T;
// C <= HT_MAX_CLASSES), and loss = sa * sum(la) + sb * sum(lb) (fixed order).
constexpr int HT_MAX_CLASSES = 64;
void ht_launch_cos(cudaStream_t st, const float* stv, const float* tgt, int n, int D, float* lossr, float* dxh);
void ht_launch_cls(cudaStream_t st, int dt, const float* zp, int n_cls, int D, const void* wc, const float* bc, int C,
                   const int* label, float scale, float* lossc, void* dpt, unsigned* err);
void ht_launch_loss(cudaStream_t st, const float* la, int na, float sa, const float* lb, int nb, float sb,
                    float* loss);
// dxh: nsplit partial sums [n][D], split_stride floats apart.
void ht_launch_out_bwd(cudaStream_t st, int dt, const float* dxh, int nsplit, size_t split_stride, const float* stv,
                       const float* h5, int n, int D, const float* g2, float eps, int mode, float norm_eps, float* dc0,
                       float* dh5f, void* dh5t, float* r2);
void ht_launch_mid_bwd(cudaStream_t st, int dt, const float* dh4, const float* h3, int n, int m1, const float* g1,
                       float eps, float* dh3f, void* dh3t, float* r1);
// GELU (bwd = 0: h = GELU(z) into hf (optional), ht, hT) or its derivative (bwd = 1: dz = hf *
// GELU'(z) in place in hf, and into ht, hT), with the transposed copy hT [C][ldT] (zero columns
// n..ldT-1) written by the same launch.
// bwd = 1 also leaves the chunk partials of the column sums of dz in part ([chunks(n)][C], for
// ht_launch_colsum_finish).
void ht_launch_gelu_tile(cudaStream_t st, int dt, int bwd, const float* z, float* hf, int n, int C, void* ht, void* hT,
                         int ldT, float* part);
void ht_launch_prep_bwd(cudaStream_t st, const float* hs, const float* hp, const float* hI, const float* dc0, int n,
                        int D, const float* g0, const float* conv, float eps, float* pg0, float* cw);
// Two launches; part holds chunks(J.n) * sum(C) floats.  Returns the launch count.
int ht_launch_colsum(cudaStream_t st, ColJobs J, float* part);
// The second half of ht_launch_colsum, for partials a producer already wrote ([chunks(J.n)][sum C]).
int ht_launch_colsum_finish(cudaStream_t st, ColJobs J, const float* part);
// dst [C][ldT] = src [n][C] transposed, zero columns n..ldT-1.
void ht_launch_transpose(cudaStream_t st, int dt, const void* src, int n, int C, void* dst, int ldT);
void ht_launch_adamw(cudaStream_t st, int dt, AdamArgs A);

}  // namespace adept
