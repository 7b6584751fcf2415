// CE-MoE layout tools (host only): the layer-composition rule of Sec. 4.1 and
// the phased-greedy layer pattern of Algorithm 1 (Sec. 4.2).  They decide how
// many routed MoE layers a hybrid model has and where they sit, i.e. the L_E
// factor of Eq. 1 that the layer kernels of this library are multiplied by.
#include <cmath>
#include <string>
#include <vector>

#include "moe.h"

namespace {

// A virtual block (m, 1_e, 1_a, 1_d): m Mamba blocks, then optional MoE,
// attention and dense-FFN blocks.
struct VBlock {
  int m;
  bool e, a, d;
  char kind;  // 'A' attention-bearing, 'N' regular, 'R' residue
};

// Mamba spine with the MoE block after floor(m / 2) Mamba blocks, attention at
// the token-mixing tail, the dense FFN last.
std::string render(const VBlock& v) {
  std::string s;
  const int before = v.e ? v.m / 2 : v.m;
  s.append(before, 'M');
  if (v.e) {
    s.push_back('E');
    s.append(v.m - before, 'M');
  }
  if (v.a) s.push_back('*');
  if (v.d) s.push_back('-');
  return s;
}

int write_out(const std::string& s, char* buf, size_t cap) {
  if (!buf) return MOE_ERR_NULL;
  if (s.size() + 1 > cap) return MOE_ERR_SHAPE;
  s.copy(buf, s.size());
  buf[s.size()] = '\0';
  return MOE_OK;
}

}  // namespace

extern "C" int moe_ce_composition(int32_t a_star, int32_t b_star, int32_t c_star, double alpha, int32_t* a,
                                  int32_t* b, int32_t* c, int32_t* d) {
  if (!a || !b || !c || !d) return MOE_ERR_NULL;
  if (a_star < 0 || b_star < 0 || c_star < 0 || !(alpha > -2.0)) return MOE_ERR_SHAPE;
  const int32_t L = a_star + b_star + c_star;
  // b = floor(L / (alpha + 2)), d = b, c = c*, the rest Mamba (Sec. 4.1)
  const int32_t nb = (int32_t)std::floor((double)L / (alpha + 2.0));
  const int32_t na = L - 2 * nb - c_star;
  if (na < 0) return MOE_ERR_SHAPE;
  *a = na;
  *b = nb;
  *c = c_star;
  *d = nb;
  return MOE_OK;
}

extern "C" int moe_ce_layer_pattern(int32_t a, int32_t b, int32_t c, int32_t d, char* pattern, size_t pattern_cap,
                                    char* blocks, size_t blocks_cap, char* decorated, size_t decorated_cap) {
  if (a < 0 || b < 0 || c < 0 || d < 0 || b < c) return MOE_ERR_SHAPE;
  int nM = a, nE = b, nA = c, nD = d;
  const int nvb = std::max(std::max(nE, nA), std::max(nD, 1));
  const int ell = (nM + nvb - 1) / nvb;  // ceil(n_M / n_vb)
  std::vector<VBlock> A, N, R;
  // Phase 1: attention-bearing blocks, each with the nominal Mamba budget
  while (nA > 0 && nM >= ell) {
    const bool e = nE > 0, dd = nD > 0;
    A.push_back(VBlock{ell, e, true, dd, 'A'});
    nM -= ell;
    nE -= e;
    nA -= 1;
    nD -= dd;
  }
  // Phase 2: regular blocks (MoE + dense FFN) with the nominal budget
  while (nM >= ell && nE > 0 && nD > 0 && ell > 0) {
    N.push_back(VBlock{ell, true, false, true, 'N'});
    nM -= ell;
    nE -= 1;
    nD -= 1;
  }
  // Phase 3: residue blocks covering what is left; one per remaining MoE,
  // attention or dense block (at least one), the remaining Mamba shared as
  // evenly as possible with the larger shares first
  if (nM + nE + nA + nD > 0) {
    const int r = std::max(std::max(nE, nA), std::max(nD, 1));
    for (int i = 0; i < r; ++i) {
      const int m = nM / r + (i < nM % r ? 1 : 0);
      R.push_back(VBlock{m, i < nE, i < nA, i < nD, 'R'});
    }
  }
  // Phase 4: the N blocks split the A sequence into |N| + 1 groups of
  // near-equal size, the larger groups first (ties broken left to right);
  // residue blocks go last
  std::vector<VBlock> order;
  const int na = (int)A.size(), nn = (int)N.size();
  const int q = na / (nn + 1), rem = na % (nn + 1);
  int ai = 0;
  for (int gidx = 0; gidx <= nn; ++gidx) {
    const int sz = q + (gidx < rem ? 1 : 0);
    for (int j = 0; j < sz; ++j) order.push_back(A[ai++]);
    if (gidx < nn) order.push_back(N[gidx]);
  }
  for (const VBlock& v : R) order.push_back(v);
  std::string pat, kinds, deco;
  for (const VBlock& v : order) {
    const std::string s = render(v);
    pat += s;
    kinds.push_back(v.kind);
    deco += (v.kind == 'A' ? "[" : "(") + s + (v.kind == 'A' ? "]" : ")");
  }
  int st = write_out(pat, pattern, pattern_cap);
  if (st != MOE_OK) return st;
  if (blocks) {
    st = write_out(kinds, blocks, blocks_cap);
    if (st != MOE_OK) return st;
  }
  if (decorated) {
    st = write_out(deco, decorated, decorated_cap);
    if (st != MOE_OK) return st;
  }
  return (int)pat.size();
}
