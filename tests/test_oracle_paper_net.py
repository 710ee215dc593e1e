"""The paper's policy network (Sec. 4.2) as the plain MLP the oracle and the kernels run.

The network: a linear projection of the 8-dim state to a 4-dim embedding, 2-head
self-attention (embedding 4) over that single token, and separate policy and value
heads (one 64-unit GELU hidden layer each).  PyTorch's own ``nn.MultiheadAttention`` and
``nn.GELU(approximate="tanh")`` modules built that way, in fp64, must give the same
logits, value, loss and parameter gradients as the oracle's MLP form
(8-4-4-4-128-34: identity, identity, identity, GELU; block-diagonal output layer),
whose weights are read off the modules.  This pins the reading that attention over one
token is the value projection followed by the output projection, and the joint-head
layout, against a library implementation rather than the oracle's own formula.
"""
import numpy as np
import pytest

from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")

N_ACT = 33


class PaperNet(torch.nn.Module):
    def __init__(self):
        super().__init__()
        self.proj = torch.nn.Linear(8, 4)
        self.attn = torch.nn.MultiheadAttention(4, 2, batch_first=True)
        self.pol = torch.nn.Sequential(torch.nn.Linear(4, 64), torch.nn.GELU(approximate="tanh"),
                                       torch.nn.Linear(64, N_ACT))
        self.val = torch.nn.Sequential(torch.nn.Linear(4, 64), torch.nn.GELU(approximate="tanh"),
                                       torch.nn.Linear(64, 1))

    def forward(self, s):
        e = self.proj(s)[:, None, :]          # one token per state
        h, _ = self.attn(e, e, e, need_weights=False)
        h = h[:, 0, :]
        return self.pol(h), self.val(h)[:, 0]


def _net(seed):
    torch.manual_seed(seed)
    net = PaperNet().double()
    with torch.no_grad():  # nonzero attention biases so every term shows
        net.attn.in_proj_bias.normal_(0.0, 0.3)
        net.attn.out_proj.bias.normal_(0.0, 0.3)
    return net


def _mlp_of(net):
    """The MLP weights (W_l [out, in], b_l) that the paper's network reduces to."""
    g = lambda t: t.detach().numpy().copy()
    ipw, ipb = g(net.attn.in_proj_weight), g(net.attn.in_proj_bias)
    W3 = np.vstack([g(net.pol[0].weight), g(net.val[0].weight)])
    b3 = np.concatenate([g(net.pol[0].bias), g(net.val[0].bias)])
    W4 = np.zeros((N_ACT + 1, 128))
    W4[:N_ACT, :64] = g(net.pol[2].weight)
    W4[N_ACT, 64:] = g(net.val[2].weight)[0]
    b4 = np.concatenate([g(net.pol[2].bias), g(net.val[2].bias)])
    Ws = [g(net.proj.weight), ipw[8:12], g(net.attn.out_proj.weight), W3, W4]
    bs = [g(net.proj.bias), ipb[8:12], g(net.attn.out_proj.bias), b3, b4]
    return Ws, bs


def _inputs(n, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, 8)) * np.array([1, 30, 5, 1, 1, 100, 0.5, 2])
    return X


def test_paper_network_forward_is_the_mlp():
    net = _net(1)
    X = _inputs(257, 2)
    with torch.no_grad():
        logits, v = net(torch.tensor(X))
    Ws, bs = _mlp_of(net)
    dims, hv = W.mlp_dims("c1p")
    assert [Ws[0].shape[1]] + [w.shape[0] for w in Ws] == dims and hv
    _, out = rl.forward(Ws, bs, X, W.mlp_acts("c1p"))
    assert np.allclose(out[:, :N_ACT], logits.numpy(), rtol=1e-12, atol=1e-12)
    assert np.allclose(out[:, N_ACT], v.numpy(), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("algo", [rl.REINFORCE, rl.PPO])
def test_paper_network_gradient_is_the_mlp_gradient(algo):
    """The oracle's loss gradient on the MLP form, read at the real parameters, equals
    autograd through the attention and head modules."""
    net = _net(3 + algo)
    n = 300
    X = _inputs(n, 4)
    rng = np.random.default_rng(5)
    a = rng.integers(0, N_ACT, n)
    adv = rng.standard_normal(n) * 2.0
    ret = rng.standard_normal(n)
    Ws, bs = _mlp_of(net)
    acts = W.mlp_acts("c1p")
    _, out = rl.forward(Ws, bs, X, acts)
    z = out[:, :N_ACT]
    lp = z - z.max(1, keepdims=True)
    lp = lp - np.log(np.exp(lp).sum(1, keepdims=True))
    lpo = lp[np.arange(n), a] + rng.choice([0.0, 0.4, -0.4], n)
    grads, stats = rl.loss_grad(Ws, bs, True, X, a, lpo, adv, ret, algo, 0.2, 0.5, 0.01, acts)

    logits, v = net(torch.tensor(X))
    logpi = torch.log_softmax(logits, 1)
    lpa = logpi[torch.arange(n), torch.tensor(a)]
    advt = torch.tensor(adv)
    if algo == rl.REINFORCE:
        pg = -(advt * lpa).mean()
    else:
        rho = torch.exp(lpa - torch.tensor(lpo))
        pg = -torch.minimum(rho * advt, torch.clamp(rho, 0.8, 1.2) * advt).mean()
    ent = -(logpi.exp() * logpi).sum(1).mean()
    loss = pg - 0.01 * ent + 0.5 * ((v - torch.tensor(ret)) ** 2).mean()
    loss.backward()
    assert stats[0] == pytest.approx(loss.item(), rel=1e-12)

    gd = lambda t: t.grad.numpy()
    ipw, ipb = gd(net.attn.in_proj_weight), gd(net.attn.in_proj_bias)
    # query and key projections do not reach the output of one-token attention
    assert np.abs(ipw[:8]).max() < 1e-12 and np.abs(ipb[:8]).max() < 1e-12
    close = lambda x, y: np.allclose(x, y, rtol=1e-9, atol=1e-12)
    (g0, c0), (g1, c1), (g2, c2), (g3, c3), (g4, c4) = grads
    assert close(g0, gd(net.proj.weight)) and close(c0, gd(net.proj.bias))
    assert close(g1, ipw[8:12]) and close(c1, ipb[8:12])
    assert close(g2, gd(net.attn.out_proj.weight)) and close(c2, gd(net.attn.out_proj.bias))
    assert close(g3[:64], gd(net.pol[0].weight)) and close(g3[64:], gd(net.val[0].weight))
    assert close(c3, np.concatenate([gd(net.pol[0].bias), gd(net.val[0].bias)]))
    assert close(g4[:N_ACT, :64], gd(net.pol[2].weight))
    assert close(g4[N_ACT, 64:], gd(net.val[2].weight)[0])
    assert close(c4, np.concatenate([gd(net.pol[2].bias), gd(net.val[2].bias)]))


def test_policy_weights_are_block_diagonal():
    dims, _ = W.mlp_dims("c1p")
    Ws, bs = W.policy_weights("c1p", dims, 9)
    assert np.all(Ws[-1][:N_ACT, 64:] == 0) and np.all(Ws[-1][N_ACT, :64] == 0)
    assert np.all(Ws[-1][:N_ACT, :64] != 0) and np.all(Ws[-1][N_ACT, 64:] != 0)
    assert all(w.dtype == np.float32 for w in Ws + bs)
