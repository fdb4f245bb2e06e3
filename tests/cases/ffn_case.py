"""Small case for an ncu capture of the fused one-token FFN: l4e64 shape, 1 layer, 22 slots."""
import sys
sys.path[:0] = [".", "tests"]
import torch, synth
from mfharness import Ctx, Shape
import paper_2607_09686_gb300 as mf
cfg = synth.CONFIGS["l4e64"]
shape = Shape(1, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype)
ctx = Ctx(shape, 22, max_tokens=1, workers=16)
T = 8
x = torch.from_numpy(synth.activations(0, 0, 0, 0, T, cfg.hidden)).cuda()
r = synth.routes(0, 0, 0, 64, 8, T, 1.1, 0.6)
b = torch.from_numpy(synth.plant_bias(r, 64)).cuda()
y = torch.empty(T, cfg.hidden, device="cuda")
for t in range(T):
    mf.mf_moe_forward(ctx.h, 0, x[t], ctx.wr[0], b[t], 1, y[t])
torch.cuda.synchronize()
assert mf.mf_check(ctx.h) == 0
print("ok")
ctx.close()
